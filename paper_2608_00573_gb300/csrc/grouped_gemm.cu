// Kernel (c): grouped expert-FFN GEMM on the 5th-generation tensor cores.
//
// For every group g (an expert, or the shared expert) with rows
// [goff[g], goff[g+1]) of the compacted activations A (bf16, K contiguous) and
// that group's weights B (bf16 [N][K], K contiguous):
//     out[row, :] = epilogue(A[row, :] . B^T)
// with epilogue = store (down projection), SwiGLU over the interleaved
// gate/up columns (W13 of a SwiGLU expert), ReLU (W1 of a ReLU expert), a
// residual add (bf16 residual row + accumulator: the attention output
// projection of the full block) or the rotary embedding of the query and key
// heads (the q/k/v projection of the full block).
// The expert FFN of the executed layers (Sec. III-B/C and the execute branch of
// Algorithm 2) is the dense contraction of the MoE step; the full block also
// runs its attention projections through this kernel as a single group.
//
// Design (one CTA per SM, persistent, 192 threads):
//   warp 0      TMA producer (one lane); also owns the TMEM allocation
//   warp 1      MMA issuer (one lane): tcgen05.mma.cta_group::1.kind::f16,
//               M = 128, N = 256, K = 16 per instruction, fp32 accumulators in
//               TMEM, two 256-column accumulators so the epilogue of one tile
//               overlaps the main loop of the next
//   warps 2-5   epilogue: tcgen05.ld 32 rows x 32 columns per warp, fused
//               activation, bf16 stores
// Operand tiles (A 128x64, B 256x64 per stage, 4 stages) arrive by TMA with
// 128-byte swizzle.  Tiles are ordered expert-major, then by blocks of row
// tiles (about 48 MB of activations), then output-column tile, then row tile,
// so concurrent CTAs share one weight tile through L2 and a block's
// activations stay resident while the weights stream.
// Every mbarrier wait is bounded (2 s); on expiry the kernel records an error
// word, stops issuing work, frees its TMEM and returns.
//
// Pair variant (launches whose groups are large): clusters of two CTAs on two
// SMs issue tcgen05.mma.cta_group::2 with M = 256, N = 256.  Each CTA stages
// its own 128 rows of A and its own half (128 output columns) of B, 32 KB per
// stage in 6 stages, and holds its 128 rows x 256 columns of the accumulator
// in its own TMEM; the even CTA issues the MMAs for both.  Per SM this halves
// the B bytes staged per FLOP, so the same shared memory keeps 5 stages
// (~2500 tensor cycles) of loads in flight instead of 3.  A row-pair tile
// covers 256 rows of one group (the odd CTA's rows may lie past the group:
// loaded, computed and masked).
//
// Transposed pair variant (routed down projections, ReLU up projections): the
// weights on the MMA's M side and the tokens on its N side, N rounded up to 16
// per tile, so a group's tail pads at most 15 tokens; described at the kernel.
//
// Both pair variants take their tiles in the order above; for long K they
// draw them from a launch-wide counter (PairTiles) rather than each cluster
// walking a fixed stride, so clusters that finish early take more tiles and
// the tiles in flight stay neighbours in that order.
#include <algorithm>

#include <climits>

#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int A_BYTES = BM * BK * 2;
constexpr int B_BYTES = BN * BK * 2;
constexpr int STAGE_BYTES = A_BYTES + B_BYTES;
constexpr int P_STAGES = 6;                       // pair variant
constexpr int PB_BYTES = (BN / 2) * BK * 2;        // this CTA's half of the B tile
constexpr int P_STAGE_BYTES = A_BYTES + PB_BYTES;
constexpr int kThreads = 192;
constexpr uint32_t TMEM_COLS = 512;
constexpr int kMaxGroups = kMaxE + 1;

constexpr int kTQ = 4;                            // tile queue depth (CTA-pair kernels)

template <int NST>
struct __align__(8) SmemTail {
    uint64_t full[NST];
    uint64_t empty[NST];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t tq_full[kTQ];         // CTA-pair kernels: tile index published (each CTA)
    uint64_t tq_empty[kTQ];        // ... and taken by every role of both CTAs (even CTA)
    int tq[kTQ];
    uint32_t tmem_base;
    int abort_flag;
    int total_tiles;
    int tile_start[kMaxGroups + 1];
    int gstart[kMaxGroups];
    int gcnt[kMaxGroups];
};
using GemmSmemTail = SmemTail<STAGES>;
using PairSmemTail = SmemTail<P_STAGES>;

constexpr size_t kSmemBytes = 1024 + (size_t)STAGES * STAGE_BYTES + sizeof(GemmSmemTail);
constexpr size_t kPairSmemBytes = 1024 + (size_t)P_STAGES * P_STAGE_BYTES + sizeof(PairSmemTail);

struct Tile {
    int rows, a_row, out_row, b_row, nt;
};

// Per-group tile counts from the device-side group offsets (tile_rows rows per
// row tile); one warp: 32 groups' offsets loaded at once, tile counts
// prefix-summed with shuffles (integer sums, the same table as a serial loop).
template <class Tail>
__device__ __forceinline__ void build_tile_table(Tail* tl, const int* goff, int first_group, int ngroups,
                                                 int n_tiles_n, int tile_rows, int lane) {
    int carry = 0;
    for (int g0 = 0; g0 < ngroups; g0 += 32) {
        const int g = g0 + lane;
        int st = 0, cnt = 0, nt = 0;
        if (g < ngroups) {
            st = goff[first_group + g];
            cnt = goff[first_group + g + 1] - st;
            nt = ((cnt + tile_rows - 1) / tile_rows) * n_tiles_n;
        }
        int incl = nt;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (g < ngroups) {
            tl->gstart[g] = st;
            tl->gcnt[g] = cnt;
            tl->tile_start[g] = carry + incl - nt;
        }
        carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) {
        tl->tile_start[ngroups] = carry;
        tl->total_tiles = carry;
        tl->abort_flag = 0;
    }
}

// Tile t -> (group, row tile, column tile).  Within a group the row tiles are
// taken in blocks of mblk (an activation block small enough to stay in L2);
// inside a block the column tile is the slow index and the row tile the fast
// one, so the CTAs running at the same time share one weight tile and the
// block's activation rows are read from HBM once.  A row tile has tile_rows
// rows; this CTA takes the 128 from sub_row on and B rows from b_sub on.
template <class Tail>
__device__ __forceinline__ void locate_tile(const Tail* tl, int t, int ngroups, int n_tiles_n, int mblk,
                                            int tile_rows, int& g, int& mt, int& nt) {
    int lo = 0, hi = ngroups - 1;
    while (lo < hi) {                      // largest g with tile_start[g] <= t
        const int mid = (lo + hi + 1) >> 1;
        if (tl->tile_start[mid] <= t) lo = mid; else hi = mid - 1;
    }
    g = lo;
    const int cnt = tl->gcnt[g];
    const int mtc = (cnt + tile_rows - 1) / tile_rows;
    const int u = t - tl->tile_start[g];
    const int nfull = mtc / mblk;
    const int full_tiles = nfull * mblk * n_tiles_n;
    if (u < full_tiles) {
        const int b = u / (mblk * n_tiles_n);
        const int r = u - b * (mblk * n_tiles_n);
        nt = r / mblk;
        mt = b * mblk + (r - nt * mblk);
    } else {
        const int last = mtc - nfull * mblk;
        const int r = u - full_tiles;
        nt = r / last;
        mt = nfull * mblk + (r - nt * last);
    }
}

template <class Tail>
__device__ __forceinline__ Tile map_tile(const Tail* tl, int t, int ngroups, int n_tiles_n, int base0,
                                         int a_rebase, int out_rebase, int b_rows_per_group, int mblk,
                                         int tile_rows, int sub_row, int b_sub) {
    int g, mt, nt;
    locate_tile(tl, t, ngroups, n_tiles_n, mblk, tile_rows, g, mt, nt);
    const int cnt = tl->gcnt[g];
    const int r0 = mt * tile_rows + sub_row;
    Tile r;
    r.rows = max(0, min(BM, cnt - r0));
    r.a_row = tl->gstart[g] - (a_rebase ? base0 : 0) + r0;
    r.out_row = tl->gstart[g] - (out_rebase ? base0 : 0) + r0;
    r.b_row = g * b_rows_per_group + nt * BN + b_sub;
    r.nt = nt;
    return r;
}

__device__ __forceinline__ void store_row32(__nv_bfloat16* dst, const float (&v)[32]) {
    uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        uint4 u;
        u.x = pack_bf16x2(v[8 * q + 0], v[8 * q + 1]);
        u.y = pack_bf16x2(v[8 * q + 2], v[8 * q + 3]);
        u.z = pack_bf16x2(v[8 * q + 4], v[8 * q + 5]);
        u.w = pack_bf16x2(v[8 * q + 6], v[8 * q + 7]);
        d4[q] = u;
    }
}

// Epilogue of one tile for one warp: TMEM lane quarter q (rows q*32 + lane),
// all BN accumulator columns at tb; K range kr when the K dimension is split.
__device__ __forceinline__ void epilogue_tile(uint32_t tb, int row, const Tile& ti, int kr, int ksplit,
                                              int epi_mode, __nv_bfloat16* __restrict__ out, int ldo,
                                              const __nv_bfloat16* __restrict__ res, int ldr,
                                              const RopeEpi& rp, float* __restrict__ partial, int ldp,
                                              size_t pstride) {
    const bool valid = row < ti.rows;
    __nv_bfloat16* orow = out + (size_t)(ti.out_row + (valid ? row : 0)) * ldo;
    if (ksplit > 1) {
        // fp32 partial sums of this K range; the finish kernel adds the ranges.
        float* prow = partial + (size_t)kr * pstride + (size_t)(ti.out_row + (valid ? row : 0)) * ldp +
                      ti.nt * BN;
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
            uint32_t r[32];
            tmem_ld_32x32(tb + c, r);
            tmem_ld_wait();
            if (valid) {
                float4* d4 = reinterpret_cast<float4*>(prow + c);
#pragma unroll
                for (int q4 = 0; q4 < 8; ++q4)
                    d4[q4] = make_float4(__uint_as_float(r[4 * q4]), __uint_as_float(r[4 * q4 + 1]),
                                         __uint_as_float(r[4 * q4 + 2]), __uint_as_float(r[4 * q4 + 3]));
            }
        }
    } else if (epi_mode == EPI_SWIGLU) {
#pragma unroll 1
        for (int c = 0; c < BN / 2; c += 32) {
            uint32_t gr[32], ur[32];
            tmem_ld_32x32(tb + c, gr);
            tmem_ld_32x32(tb + BN / 2 + c, ur);
            tmem_ld_wait();
            if (valid) {
                float v[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float gt = __uint_as_float(gr[i]);
                    const float up = __uint_as_float(ur[i]);
                    v[i] = gt / (1.f + __expf(-gt)) * up;
                }
                store_row32(orow + ti.nt * (BN / 2) + c, v);
            }
        }
    } else if (epi_mode == EPI_ROPE) {
        // Rotary embedding of the query and key heads in the leading n_rot
        // columns (pairs i, i + Dh/2 of each head; position = row mod S),
        // the remaining (value) heads stored as they are.
        const int tok = ti.out_row + (valid ? row : 0);
        const int pos = tok % rp.S;
        const int half = rp.dh >> 1;
#pragma unroll 1
        for (int h0 = 0; h0 < BN; h0 += rp.dh) {
            const int col0 = ti.nt * BN + h0;
            if (col0 < rp.n_rot) {
#pragma unroll 1
                for (int c = 0; c < half; c += 32) {
                    uint32_t xa[32], xb[32];
                    tmem_ld_32x32(tb + h0 + c, xa);
                    tmem_ld_32x32(tb + h0 + half + c, xb);
                    tmem_ld_wait();
                    if (valid) {
                        const float2* cs = rp.cs + (size_t)pos * half + c;
                        float ya[32], yb[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            const float2 w = __ldg(cs + i);
                            const float x1 = __uint_as_float(xa[i]), x2 = __uint_as_float(xb[i]);
                            ya[i] = x1 * w.x - x2 * w.y;
                            yb[i] = x2 * w.x + x1 * w.y;
                        }
                        store_row32(orow + col0 + c, ya);
                        store_row32(orow + col0 + half + c, yb);
                    }
                }
            } else if (rp.vt) {
                // Value heads, transposed per sequence: for each feature the
                // warp's 32 tokens are 32 consecutive key slots (64-byte stores).
                const int seq = tok / rp.S;
                __nv_bfloat16* vcol =
                    rp.vt + ((size_t)seq * rp.vt_rows + (col0 - rp.n_rot)) * kVtSlots + (tok - seq * rp.S);
#pragma unroll 1
                for (int c = 0; c < rp.dh; c += 32) {
                    uint32_t r[32];
                    tmem_ld_32x32(tb + h0 + c, r);
                    tmem_ld_wait();
                    if (valid) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            vcol[(size_t)(c + i) * kVtSlots] = __float2bfloat16_rn(__uint_as_float(r[i]));
                    }
                }
            } else {
#pragma unroll 1
                for (int c = 0; c < rp.dh; c += 32) {
                    uint32_t r[32];
                    tmem_ld_32x32(tb + h0 + c, r);
                    tmem_ld_wait();
                    if (valid) {
                        float v[32];
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
                        store_row32(orow + col0 + c, v);
                    }
                }
            }
        }
    } else {
#pragma unroll 1
        for (int c = 0; c < BN; c += 32) {
            uint32_t r[32];
            tmem_ld_32x32(tb + c, r);
            tmem_ld_wait();
            if (valid) {
                float v[32];
#pragma unroll
                for (int i = 0; i < 32; ++i) {
                    const float x = __uint_as_float(r[i]);
                    v[i] = epi_mode == EPI_RELU ? fmaxf(x, 0.f) : x;
                }
                if (epi_mode == EPI_RESID) {
                    const uint4* rr = reinterpret_cast<const uint4*>(
                        res + (size_t)(ti.out_row + row) * ldr + ti.nt * BN + c);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const uint4 w = __ldg(rr + q4);
                        v[q4 * 8 + 0] += bf16_lo(w.x);
                        v[q4 * 8 + 1] += bf16_hi(w.x);
                        v[q4 * 8 + 2] += bf16_lo(w.y);
                        v[q4 * 8 + 3] += bf16_hi(w.y);
                        v[q4 * 8 + 4] += bf16_lo(w.z);
                        v[q4 * 8 + 5] += bf16_hi(w.z);
                        v[q4 * 8 + 6] += bf16_lo(w.w);
                        v[q4 * 8 + 7] += bf16_hi(w.w);
                    }
                }
                store_row32(orow + ti.nt * BN + c, v);
            }
        }
    }
}
__global__ void __launch_bounds__(kThreads, 1)
grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const int* __restrict__ goff, int first_group, int ngroups, int a_rebase,
                    int out_rebase, int K, int n_tiles_n, int b_rows_per_group, int epi_mode,
                    __nv_bfloat16* __restrict__ out, int ldo, int* err,
                    const __nv_bfloat16* __restrict__ res, int ldr, const RopeEpi rp,
                    int mblk, int ksplit, float* __restrict__ partial,
                    int ldp, size_t pstride) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    const uint32_t pad = ((raw_addr + 1023u) & ~1023u) - raw_addr;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sA = smem_u32(smem);
    const uint32_t sB = sA + STAGES * A_BYTES;
    GemmSmemTail* tl = reinterpret_cast<GemmSmemTail*>(smem + (size_t)STAGES * STAGE_BYTES);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    // Set-up that touches only this CTA's own resources (barriers, TMEM,
    // descriptor prefetch) runs before the programmatic wait, under the
    // preceding kernel's tail.
    if (threadIdx.x == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(smem_u32(&tl->full[s]), 1);
            mbar_init(smem_u32(&tl->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&tl->tfull[b]), 1);
            mbar_init(smem_u32(&tl->tempty[b]), 4);
        }
        fence_barrier_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
    }
    if (warp == 0) tmem_alloc(smem_u32(&tl->tmem_base), TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = tl->tmem_base;
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now

    // Tile table from the device-side group offsets.
    if (warp == 0) build_tile_table(tl, goff, first_group, ngroups, n_tiles_n, BM, lane);
    __syncthreads();
    const int ntiles = tl->total_tiles;
    const int total = ntiles * ksplit;    // unit u: tile u % ntiles, K range u / ntiles
    if ((int)blockIdx.x >= total) {
        if (warp == 0) {
            __syncwarp();
            tc_fence_after();
            tmem_dealloc(tmem_base, TMEM_COLS);
        }
        return;
    }
    const int base0 = tl->gstart[0];
    const int nkb = K / BK;
    const int kbr = nkb / ksplit;         // k blocks per range
    volatile int* abort_flag = &tl->abort_flag;

    if (warp == 0) {
        if (lane == 0) {
            // ---------------------------------------------------- producer
            int it = 0;
            for (int t = blockIdx.x; t < total && !*abort_flag; t += gridDim.x) {
                const Tile ti = map_tile(tl, t % ntiles, ngroups, n_tiles_n, base0, a_rebase, out_rebase,
                                         b_rows_per_group, mblk, BM, 0, 0);
                const int kb0 = (t / ntiles) * kbr;
                for (int kb = kb0; kb < kb0 + kbr; ++kb, ++it) {
                    const int s = it % STAGES;
                    const uint32_t ph = (it / STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->empty[s]), ph ^ 1, abort_flag, err,
                                           ERR_TIMEOUT_PRODUCER))
                        break;
                    const uint32_t fb = smem_u32(&tl->full[s]);
                    mbar_arrive_expect_tx(fb, STAGE_BYTES);
                    tma_load_2d(sA + s * A_BYTES, &tmA, kb * BK, ti.a_row, fb);
                    tma_load_2d(sB + s * B_BYTES, &tmB, kb * BK, ti.b_row, fb);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------------------------------------------- MMA issuer
            constexpr uint32_t idesc = idesc_bf16_f32(BM, BN);
            int it = 0, tl_i = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < total && ok; t += gridDim.x, ++tl_i) {
                const int buf = tl_i & 1;
                const uint32_t aph = (tl_i >> 1) & 1;
                if (!mbar_wait_bounded(smem_u32(&tl->tempty[buf]), aph ^ 1, abort_flag, err,
                                       ERR_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                const int kb0 = (t / ntiles) * kbr;
                for (int kb = kb0; kb < kb0 + kbr; ++kb, ++it) {
                    const int s = it % STAGES;
                    const uint32_t ph = (it / STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->full[s]), ph, abort_flag, err, ERR_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = sA + s * A_BYTES;
                    const uint32_t b0 = sB + s * B_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        tc_mma_bf16(d_tmem, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32),
                                    idesc, (kb != kb0 || kk != 0) ? 1u : 0u);
                    tc_commit(smem_u32(&tl->empty[s]));
                }
                if (!ok) break;
                tc_commit(smem_u32(&tl->tfull[buf]));
            }
        }
    } else {
        // -------------------------------------------------------- epilogue
        const int q = warp & 3;                 // TMEM lane quarter of this warp
        const int row = q * 32 + lane;
        int tl_i = 0;
        for (int t = blockIdx.x; t < total; t += gridDim.x, ++tl_i) {
            const Tile ti = map_tile(tl, t % ntiles, ngroups, n_tiles_n, base0, a_rebase, out_rebase,
                                     b_rows_per_group, mblk, BM, 0, 0);
            const int buf = tl_i & 1;
            const uint32_t aph = (tl_i >> 1) & 1;
            int ok = 1;
            if (lane == 0)
                ok = mbar_wait_bounded(smem_u32(&tl->tfull[buf]), aph, abort_flag, err, ERR_TIMEOUT_EPI);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN);
            epilogue_tile(tb, row, ti, t / ntiles, ksplit, epi_mode, out, ldo, res, ldr, rp, partial, ldp,
                          pstride);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&tl->tempty[buf]));
        }
    }

    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

// Tile sequence of a CTA pair.  Its first tile is cid; after that the even
// CTA's producer draws the next tile index from a launch-wide counter (tiles
// in order, so the tiles in flight stay neighbours in the L2-blocked order,
// and a pair whose tiles ran short takes more of them), one draw ahead so that
// the atomic's latency hides behind the current tile's loads, and publishes
// each index to both CTAs through a queue of kTQ slots (tq_full in each CTA,
// tq_empty in the even CTA counting the ten roles that take every entry: the
// odd CTA's producer, the MMA issuer, and both CTAs' four epilogue warps).
// Without a counter every role walks the static order cid, cid + ncl, ... on
// its own.  An index >= the tile count ends the sequence.
template <class Tail>
struct PairTiles {
    Tail* tl;
    int* sched;
    int cid, ncl;
    uint32_t rank;
    volatile int* abort_flag;
    int* err;

    __device__ __forceinline__ int draw(int i) const {       // the pair's tile for step i >= 1
        return sched ? ncl + atomicAdd(sched, 1) : cid + i * ncl;
    }
    // Even CTA's producer: publish tile t as step i (INT_MAX if a wait gave up).
    __device__ __forceinline__ int publish(int i, int t) const {
        const int slot = i % kTQ;
        if (i >= kTQ && !mbar_wait_bounded(smem_u32(&tl->tq_empty[slot]), ((i / kTQ) - 1) & 1, abort_flag, err,
                                           ERR_TIMEOUT_PRODUCER))
            return INT_MAX;
        tl->tq[slot] = t;
        st_shared_cluster_u32(mapa_shared(smem_u32(&tl->tq[slot]), 1), (uint32_t)t);
        mbar_arrive(smem_u32(&tl->tq_full[slot]));
        mbar_arrive_cluster(mapa_shared(smem_u32(&tl->tq_full[slot]), 1));
        return t;
    }
    // Every other role (one thread each): the tile of step i.
    __device__ __forceinline__ int take(int i, int code) const {
        if (!sched) return cid + i * ncl;
        const int slot = i % kTQ;
        if (!mbar_wait_bounded(smem_u32(&tl->tq_full[slot]), (i / kTQ) & 1, abort_flag, err, code)) return INT_MAX;
        const int t = *reinterpret_cast<volatile int*>(&tl->tq[slot]);
        if (rank == 0) mbar_arrive(smem_u32(&tl->tq_empty[slot]));
        else mbar_arrive_cluster(mapa_shared(smem_u32(&tl->tq_empty[slot]), 0));
        return t;
    }
    // Producer of either CTA: the tile of step i; t_next carries the even
    // CTA's draw for the next step.
    __device__ __forceinline__ int producer_step(int i, int ntiles, int& t_next) const {
        if (!sched) return cid + i * ncl;
        if (rank != 0) return take(i, ERR_TIMEOUT_PRODUCER);
        const int t = publish(i, t_next);
        if (t < ntiles) t_next = draw(i + 1);
        return t;
    }
};

__device__ __forceinline__ void init_tile_queue_bars(uint64_t* tq_full, uint64_t* tq_empty) {
    for (int b = 0; b < kTQ; ++b) {
        mbar_init(smem_u32(&tq_full[b]), 1);
        mbar_init(smem_u32(&tq_empty[b]), 10);
    }
}

// Pair variant: one cluster of two CTAs per row-pair tile of 256 rows x 256
// columns.  The tile sequence is shared by both CTAs; CTA rank r takes rows
// [r * 128, r * 128 + 128) of the tile and B rows (output columns)
// [r * 128, r * 128 + 128) of the column tile.
//   full[s]   (even CTA)  both CTAs' TMA loads of stage s complete on it
//   empty[s]  (each CTA)  released by the even CTA's MMA commit, multicast
//   tfull[b]  (each CTA)  accumulator b ready, multicast commit
//   tempty[b] (even CTA)  8 arrivals: the 4 epilogue warps of each CTA
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
grouped_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                         const int* __restrict__ goff, int first_group, int ngroups, int a_rebase,
                         int out_rebase, int K, int n_tiles_n, int b_rows_per_group, int epi_mode,
                         __nv_bfloat16* __restrict__ out, int ldo, int* err,
                         const __nv_bfloat16* __restrict__ res, int ldr, const RopeEpi rp, int mblk,
                         int* __restrict__ sched) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    const uint32_t pad = ((raw_addr + 1023u) & ~1023u) - raw_addr;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sA = smem_u32(smem);
    const uint32_t sB = sA + P_STAGES * A_BYTES;
    PairSmemTail* tl = reinterpret_cast<PairSmemTail*>(smem + (size_t)P_STAGES * P_STAGE_BYTES);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();      // 0: issues the MMAs, 1: peer
    const int cid = (int)(blockIdx.x >> 1), ncl = (int)(gridDim.x >> 1);
    const int sub = (int)rank * (BM);             // this CTA's rows / B rows within the tile

    // Set-up that touches only the pair's own resources runs before the
    // programmatic wait, under the preceding kernel's tail.
    if (threadIdx.x == 0) {
        for (int s = 0; s < P_STAGES; ++s) {
            mbar_init(smem_u32(&tl->full[s]), 1);
            mbar_init(smem_u32(&tl->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&tl->tfull[b]), 1);
            mbar_init(smem_u32(&tl->tempty[b]), 8);
        }
        init_tile_queue_bars(tl->tq_full, tl->tq_empty);
        fence_barrier_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmB);
    }
    if (warp == 0) tmem_alloc_pair(smem_u32(&tl->tmem_base), TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    cluster_sync();                               // both CTAs' barriers are initialised
    tc_fence_after();
    const uint32_t tmem_base = tl->tmem_base;
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now

    if (warp == 0) build_tile_table(tl, goff, first_group, ngroups, n_tiles_n, 2 * BM, lane);
    __syncthreads();
    const int ntiles = tl->total_tiles;
    const int base0 = tl->gstart[0];
    const int nkb = K / BK;
    volatile int* abort_flag = &tl->abort_flag;
    const PairTiles<PairSmemTail> tiles{tl, sched, cid, ncl, rank, abort_flag, err};

    if (warp == 0) {
        if (lane == 0) {
            // ---------------------------------------------------- producer (both CTAs)
            int it = 0;
            int t_next = cid;
            for (int i = 0; !*abort_flag; ++i) {
                const int t = tiles.producer_step(i, ntiles, t_next);
                if (t >= ntiles) break;
                const Tile ti = map_tile(tl, t, ngroups, n_tiles_n, base0, a_rebase, out_rebase,
                                         b_rows_per_group, mblk, 2 * BM, sub, sub);
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % P_STAGES;
                    const uint32_t ph = (it / P_STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->empty[s]), ph ^ 1, abort_flag, err,
                                           ERR_TIMEOUT_PRODUCER))
                        break;
                    if (rank == 0) mbar_arrive_expect_tx(smem_u32(&tl->full[s]), 2 * P_STAGE_BYTES);
                    const uint32_t fb = mapa_shared(smem_u32(&tl->full[s]), 0);
                    tma_load_2d_pair(sA + s * A_BYTES, &tmA, kb * BK, ti.a_row, fb);
                    tma_load_2d_pair(sB + s * PB_BYTES, &tmB, kb * BK, ti.b_row, fb);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ---------------------------------------------------- MMA issuer (even CTA)
            constexpr uint32_t idesc = idesc_bf16_f32(2 * BM, BN);
            int it = 0, tl_i = 0;
            bool ok = true;
            for (; ok; ++tl_i) {
                if (tiles.take(tl_i, ERR_TIMEOUT_MMA) >= ntiles) break;
                const int buf = tl_i & 1;
                const uint32_t aph = (tl_i >> 1) & 1;
                if (!mbar_wait_bounded(smem_u32(&tl->tempty[buf]), aph ^ 1, abort_flag, err,
                                       ERR_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % P_STAGES;
                    const uint32_t ph = (it / P_STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->full[s]), ph, abort_flag, err, ERR_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = sA + s * A_BYTES;
                    const uint32_t b0 = sB + s * PB_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        tc_mma_bf16_pair(d_tmem, smem_desc_sw128(a0 + kk * 32), smem_desc_sw128(b0 + kk * 32),
                                         idesc, (kb != 0 || kk != 0) ? 1u : 0u);
                    tc_commit_pair_mc(smem_u32(&tl->empty[s]), 0x3);
                }
                if (!ok) break;
                tc_commit_pair_mc(smem_u32(&tl->tfull[buf]), 0x3);
            }
        }
    } else {
        // -------------------------------------------------------- epilogue (both CTAs)
        const int q = warp & 3;
        const int row = q * 32 + lane;
        int tl_i = 0;
        for (;; ++tl_i) {
            int t = 0;
            if (lane == 0) t = tiles.take(tl_i, ERR_TIMEOUT_EPI);
            t = __shfl_sync(0xffffffffu, t, 0);
            if (t >= ntiles) break;
            const Tile ti = map_tile(tl, t, ngroups, n_tiles_n, base0, a_rebase, out_rebase,
                                     b_rows_per_group, mblk, 2 * BM, sub, sub);
            const int buf = tl_i & 1;
            const uint32_t aph = (tl_i >> 1) & 1;
            int ok = 1;
            if (lane == 0)
                ok = mbar_wait_bounded(smem_u32(&tl->tfull[buf]), aph, abort_flag, err, ERR_TIMEOUT_EPI);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN);
            epilogue_tile(tb, row, ti, 0, 1, epi_mode, out, ldo, res, ldr, rp, nullptr, 0, 0);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (rank == 0) mbar_arrive(smem_u32(&tl->tempty[buf]));
                else mbar_arrive_cluster(mapa_shared(smem_u32(&tl->tempty[buf]), 0));
            }
        }
    }

    // A CTA that gave up tells its peer, so that the peer stops waiting on it.
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag)
        st_shared_cluster_u32(mapa_shared(smem_u32(&tl->abort_flag), rank ^ 1u), 1u);
    cluster_sync();                               // no access to the peer's memory remains in flight
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, TMEM_COLS);
    }
}

// ---------------------------------------------------------------------------
// Transposed pair variant (the routed experts' down projection, and the
// up projection of ReLU experts): the weights take the M side and the tokens
// the N side of tcgen05.mma.cta_group::2, D = W . X^T with M = 256 output
// features and N = the tile's tokens rounded up to 16 (at most 256).  A
// group's last token tile then computes at most 15 padded tokens, not up to
// 255 padded rows, while each SM still stages only half of the shared operand
// per FLOP.  Tiles are (group, block of token tiles, feature tile, token tile)
// in the order of map_tile.  CTA rank r stages weight rows (features)
// [r 128, r 128 + 128) of the feature tile and tokens [r N/2, (r+1) N/2) of
// the tile; its TMEM lane is an output feature and its column a token.
// Every MMA reads its operands from shared memory while TMA refills it, so
// for long K (the main loop hides the epilogue) each warp stores its 32
// features of a token straight from registers as one 64-byte segment; for
// short K the epilogue is on the critical path and the results are staged in
// shared memory and stored as 16-byte pieces of the tokens' rows.
// SwiGLU stays on the kernels above: its gate and up accumulators would sit
// in different warps' TMEM lanes, and every way of bringing them together
// that was tried (through shared memory, or 16-row weight boxes that pair
// them within a warp) was slower than the padding it saves.
constexpr int kStageBf16 = 32 * 128;           // one 32-token x 128-feature bf16 staging buffer
constexpr size_t kPairTailBytes = (sizeof(PairSmemTail) + 15) & ~(size_t)15;
constexpr size_t kPairTSmemBytes = 1024 + (size_t)P_STAGES * P_STAGE_BYTES + kPairTailBytes +
                                   2 * kStageBf16 * sizeof(__nv_bfloat16);
constexpr int kEpiBar = 1;                    // named barrier of the four epilogue warps
// Store / ReLU epilogues stage their results in shared memory up to this K
// (the launcher passes the choice as `staged`).  At K = 14336 (the
// Mixtral-shaped down projection) staged and direct stores measured the same
// forward time (196.6-198.6 vs 196.7-198.3 ms, three runs each).
constexpr int kStagedMaxK = 4096;

__device__ __forceinline__ void bar_sync_named(int id, int n) {
    asm volatile("barrier.sync %0, %1;" ::"r"(id), "r"(n) : "memory");
}

// AND of pred over the n threads of named barrier id (a barrier as well).
__device__ __forceinline__ int bar_and_named(int id, int n, int pred) {
    uint32_t r;
    asm volatile(
        "{\n\t.reg .pred p, q;\n\t"
        "setp.ne.u32 p, %1, 0;\n\t"
        "barrier.red.and.pred q, %2, %3, p;\n\t"
        "selp.u32 %0, 1, 0, q;\n\t}"
        : "=r"(r)
        : "r"(pred), "r"(id), "r"(n)
        : "memory");
    return (int)r;
}

// Token rows of tile (g, mt); the tile's MMA takes N = this rounded up to 16.
template <class Tail>
__device__ __forceinline__ int tile_tokens(const Tail* tl, int g, int mt) {
    return min(2 * BM, tl->gcnt[g] - mt * 2 * BM);
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
grouped_gemm_pair_t_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmW,
                           const int* __restrict__ goff,
                           int first_group, int ngroups, int x_rebase, int out_rebase, int K, int n_ft,
                           int w_rows_per_group, int epi_mode, __nv_bfloat16* __restrict__ out, int ldo,
                           int* err, int mblk, int staged, int* __restrict__ sched) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    const uint32_t pad = ((raw_addr + 1023u) & ~1023u) - raw_addr;
    uint8_t* smem = smem_raw + pad;
    const uint32_t sW = smem_u32(smem);                 // weight rows (M side), A_BYTES per stage
    const uint32_t sX = sW + P_STAGES * A_BYTES;        // token rows (N side), PB_BYTES per stage
    PairSmemTail* tl = reinterpret_cast<PairSmemTail*>(smem + (size_t)P_STAGES * P_STAGE_BYTES);
    uint8_t* stage_out = smem + (size_t)P_STAGES * P_STAGE_BYTES + kPairTailBytes;   // two staging buffers

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();      // 0: issues the MMAs, 1: peer
    const int cid = (int)(blockIdx.x >> 1), ncl = (int)(gridDim.x >> 1);

    // Set-up that touches only the pair's own resources runs before the
    // programmatic wait, under the preceding kernel's tail.
    if (threadIdx.x == 0) {
        for (int s = 0; s < P_STAGES; ++s) {
            mbar_init(smem_u32(&tl->full[s]), 1);
            mbar_init(smem_u32(&tl->empty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&tl->tfull[b]), 1);
            mbar_init(smem_u32(&tl->tempty[b]), 8);
        }
        init_tile_queue_bars(tl->tq_full, tl->tq_empty);
        fence_barrier_init();
        prefetch_tmap(&tmX);
        prefetch_tmap(&tmW);
    }
    if (warp == 0) tmem_alloc_pair(smem_u32(&tl->tmem_base), TMEM_COLS);
    tc_fence_before();
    __syncthreads();
    cluster_sync();                               // both CTAs' barriers are initialised
    tc_fence_after();
    const uint32_t tmem_base = tl->tmem_base;
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now

    if (warp == 0) build_tile_table(tl, goff, first_group, ngroups, n_ft, 2 * BM, lane);
    __syncthreads();
    const int ntiles = tl->total_tiles;
    const int base0 = tl->gstart[0];
    const int nkb = K / BK;
    volatile int* abort_flag = &tl->abort_flag;

    const PairTiles<PairSmemTail> tiles{tl, sched, cid, ncl, rank, abort_flag, err};

    if (warp == 0) {
        if (lane == 0) {
            // ---------------------------------------------------- producer (both CTAs)
            int it = 0;
            int t_next = cid;
            for (int i = 0; !*abort_flag; ++i) {
                const int t = tiles.producer_step(i, ntiles, t_next);
                if (t >= ntiles) break;
                int g, mt, ft;
                locate_tile(tl, t, ngroups, n_ft, mblk, 2 * BM, g, mt, ft);
                const int half = ((tile_tokens(tl, g, mt) + 15) & ~15) >> 1;
                const int xrow = tl->gstart[g] - (x_rebase ? base0 : 0) + mt * 2 * BM + (int)rank * half;
                const int wrow = g * w_rows_per_group + ft * 2 * BM;
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % P_STAGES;
                    const uint32_t ph = (it / P_STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->empty[s]), ph ^ 1, abort_flag, err,
                                           ERR_TIMEOUT_PRODUCER))
                        break;
                    if (rank == 0) mbar_arrive_expect_tx(smem_u32(&tl->full[s]), 2 * P_STAGE_BYTES);
                    const uint32_t fb = mapa_shared(smem_u32(&tl->full[s]), 0);
                    tma_load_2d_pair(sW + s * A_BYTES, &tmW, kb * BK, wrow + (int)rank * BM, fb);
                    tma_load_2d_pair(sX + s * PB_BYTES, &tmX, kb * BK, xrow, fb);
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && rank == 0) {
            // ---------------------------------------------------- MMA issuer (even CTA)
            int it = 0, tl_i = 0;
            bool ok = true;
            for (; ok; ++tl_i) {
                const int t = tiles.take(tl_i, ERR_TIMEOUT_MMA);
                if (t >= ntiles) break;
                int g, mt, ft;
                locate_tile(tl, t, ngroups, n_ft, mblk, 2 * BM, g, mt, ft);
                const uint32_t idesc = idesc_bf16_f32(2 * BM, (tile_tokens(tl, g, mt) + 15) & ~15);
                const int buf = tl_i & 1;
                const uint32_t aph = (tl_i >> 1) & 1;
                if (!mbar_wait_bounded(smem_u32(&tl->tempty[buf]), aph ^ 1, abort_flag, err,
                                       ERR_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(buf * BN);
                for (int kb = 0; kb < nkb; ++kb, ++it) {
                    const int s = it % P_STAGES;
                    const uint32_t ph = (it / P_STAGES) & 1;
                    if (!mbar_wait_bounded(smem_u32(&tl->full[s]), ph, abort_flag, err, ERR_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t w0 = sW + s * A_BYTES;
                    const uint32_t x0 = sX + s * PB_BYTES;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        tc_mma_bf16_pair(d_tmem, smem_desc_sw128(w0 + kk * 32), smem_desc_sw128(x0 + kk * 32),
                                         idesc, (kb != 0 || kk != 0) ? 1u : 0u);
                    tc_commit_pair_mc(smem_u32(&tl->empty[s]), 0x3);
                }
                if (!ok) break;
                tc_commit_pair_mc(smem_u32(&tl->tfull[buf]), 0x3);
            }
        }
    } else {
        // -------------------------------------------------------- epilogue (both CTAs)
        const int q = warp & 3;                   // TMEM lane quarter of this warp
        const int et = (warp - 2) * 32 + lane;    // epilogue thread 0..127
        int tl_i = 0, chunk = 0;
        for (;; ++tl_i) {
            int t = 0;
            if (lane == 0) t = tiles.take(tl_i, ERR_TIMEOUT_EPI);
            t = __shfl_sync(0xffffffffu, t, 0);
            // The four warps leave together (a queue wait that gave up in one
            // of them ends the others too): they meet at named barriers below.
            if (sched ? !bar_and_named(kEpiBar, 128, t < ntiles) : t >= ntiles) break;
            int g, mt, ft;
            locate_tile(tl, t, ngroups, n_ft, mblk, 2 * BM, g, mt, ft);
            const int rows = tile_tokens(tl, g, mt);
            const int nch = (((rows + 15) & ~15) + 31) / 32;
            const size_t orow = (size_t)(tl->gstart[g] - (out_rebase ? base0 : 0) + mt * 2 * BM);
            const int buf = tl_i & 1;
            const uint32_t aph = (tl_i >> 1) & 1;
            int ok = 1;
            if (lane == 0)
                ok = mbar_wait_bounded(smem_u32(&tl->tfull[buf]), aph, abort_flag, err, ERR_TIMEOUT_EPI);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            // The four warps take the same branch (they meet at named barriers below).
            if (!bar_and_named(kEpiBar, 128, ok)) break;
            tc_fence_after();
            const uint32_t tb = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(buf * BN);
            if (!staged) {
                // Long K: the main loop hides the epilogue, and shared-memory
                // traffic would compete with the MMA operand reads, so each
                // warp stores its 32 features of a token as one 64-byte segment.
                __nv_bfloat16* ocol = out + (size_t)ft * 2 * BM + (size_t)rank * BM + q * 32 + lane;
                const bool relu = epi_mode == EPI_RELU;
#pragma unroll 1
                for (int c = 0; c < nch; ++c) {
                    uint32_t r[32];
                    tmem_ld_32x32(tb + c * 32, r);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const int tok = c * 32 + j;
                        if (tok < rows) {
                            const float x = __uint_as_float(r[j]);
                            ocol[(orow + tok) * ldo] = __float2bfloat16_rn(relu ? fmaxf(x, 0.f) : x);
                        }
                    }
                }
            } else {
                // Short K: the epilogue is on the critical path; each warp
                // stages its 32 features of 32 tokens and the tokens' 256-byte
                // rows are stored as 16-byte pieces.
                __nv_bfloat16* hbase = reinterpret_cast<__nv_bfloat16*>(stage_out);
                __nv_bfloat16* ocol = out + (size_t)ft * 2 * BM + (size_t)rank * BM;
                const bool relu = epi_mode == EPI_RELU;
#pragma unroll 1
                for (int c = 0; c < nch; ++c, ++chunk) {
                    __nv_bfloat16* hb = hbase + (chunk & 1) * 32 * 128;
                    uint32_t r[32];
                    tmem_ld_32x32(tb + c * 32, r);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        const float x = __uint_as_float(r[j]);
                        hb[j * 128 + q * 32 + lane] = __float2bfloat16_rn(relu ? fmaxf(x, 0.f) : x);
                    }
                    bar_sync_named(kEpiBar, 128);
#pragma unroll
                    for (int i = et; i < 32 * 16; i += 128) {
                        const int row = i >> 4, seg = i & 15, tok = c * 32 + row;
                        if (tok < rows)
                            *reinterpret_cast<uint4*>(ocol + (orow + tok) * ldo + seg * 8) =
                                *reinterpret_cast<const uint4*>(hb + row * 128 + seg * 8);
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (rank == 0) mbar_arrive(smem_u32(&tl->tempty[buf]));
                else mbar_arrive_cluster(mapa_shared(smem_u32(&tl->tempty[buf]), 0));
            }
        }
    }

    // A CTA that gave up tells its peer, so that the peer stops waiting on it.
    __syncthreads();
    if (threadIdx.x == 0 && *abort_flag)
        st_shared_cluster_u32(mapa_shared(smem_u32(&tl->abort_flag), rank ^ 1u), 1u);
    cluster_sync();                               // no access to the peer's memory remains in flight
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, TMEM_COLS);
    }
}

}  // namespace

size_t grouped_gemm_smem_bytes() { return kSmemBytes; }

namespace {

// Clusters of two that fit on the device at once (the pair kernel is
// persistent, so it launches no more than that); 0 if none.
template <typename Kernel>
int clusters_of_two(Kernel kernel, size_t smem, int num_sms) {
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return 0;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(num_sms & ~1), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    int ncl = 0;
    if (cudaOccupancyMaxActiveClusters(&ncl, kernel, &cfg) != cudaSuccess) {
        cudaGetLastError();
        return 0;
    }
    return std::min(ncl, num_sms / 2);
}

int pair_clusters(int num_sms) {
    static PerDevice n;
    return n.get([num_sms] { return clusters_of_two(grouped_gemm_pair_kernel, kPairSmemBytes, num_sms); });
}

// The same for the transposed pair kernel (a little more shared memory).
int pair_t_clusters(int num_sms) {
    static PerDevice n;
    return n.get([num_sms] { return clusters_of_two(grouped_gemm_pair_t_kernel, kPairTSmemBytes, num_sms); });
}

}  // namespace

int grouped_gemm_pair_clusters(int num_sms) { return pair_clusters(num_sms); }

cudaError_t launch_grouped_gemm(const GemmLaunch& g, int num_sms, cudaStream_t st) {
    static PerDevice attr;
    const cudaError_t ea = (cudaError_t)attr.get([] {
        return (int)cudaFuncSetAttribute(grouped_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kSmemBytes);
    }, true);
    if (ea != cudaSuccess) return ea;
    if (g.ngroups <= 0 || g.ngroups > kMaxGroups || g.K % BK != 0) return cudaErrorInvalidValue;
    const RopeEpi rp{g.rope, g.rope_S, g.rope_dh, g.n_rot, g.vt, g.vt_rows};
    // Row tiles per block: about 48 MB of activations (a third of L2), so that
    // a block stays resident while the weight tiles stream past it.
    const long long a_tile_bytes = (long long)BM * g.K * 2;
    if (g.transposed && g.tmB_pair && g.ksplit <= 1 && pair_t_clusters(num_sms) > 0) {
        if (g.epi_mode != EPI_STORE && g.epi_mode != EPI_RELU) return cudaErrorInvalidValue;
        // Token-tile blocks of about 64 MB of activations: at K = 14336 eight
        // token tiles, so a round of 76 tiles spans ~9.5 feature tiles x 8 token
        // tiles, close to the square that streams the fewest operand slices
        // (DRAM reads of the Mixtral-shaped down launch -9 % against 32 MB).
        const int mblk2 = (int)std::max(1LL, (64LL << 20) / (2 * a_tile_bytes));
        const cudaError_t e = launch_pdl(
            grouped_gemm_pair_t_kernel, dim3(2 * pair_t_clusters(num_sms)), dim3(kThreads), kPairTSmemBytes, st,
            *g.tmA, *g.tmB_pair, g.goff, g.first_group, g.ngroups, g.a_rebase, g.out_rebase, g.K, g.n_tiles_n,
            g.b_rows_per_group, g.epi_mode, g.out, g.ldo, g.err, mblk2,
            g.K <= kStagedMaxK ? 1 : 0, g.sched);
        if (e != cudaSuccess) return e;
        return cudaGetLastError();
    }
    if (g.tmB_pair && (g.ksplit <= 1) && pair_clusters(num_sms) > 0) {
        // Row-pair tiles per block: about 32 MB of activations (same speed as
        // 40 or 48 MB within the run-to-run spread, fewest DRAM re-reads).
        const int mblk2 = (int)std::max(1LL, (32LL << 20) / (2 * a_tile_bytes));
        const cudaError_t e = launch_pdl(
            grouped_gemm_pair_kernel, dim3(2 * pair_clusters(num_sms)), dim3(kThreads), kPairSmemBytes, st, *g.tmA,
            *g.tmB_pair, g.goff, g.first_group, g.ngroups, g.a_rebase, g.out_rebase, g.K, g.n_tiles_n,
            g.b_rows_per_group, g.epi_mode, g.out, g.ldo, g.err, g.res, g.ldr, rp, mblk2, g.sched);
        if (e != cudaSuccess) return e;
        return cudaGetLastError();
    }
    const int mblk = (int)std::max(1LL, (48LL << 20) / a_tile_bytes);
    const cudaError_t e = launch_pdl(
        grouped_gemm_kernel, dim3(num_sms), dim3(kThreads), kSmemBytes, st, *g.tmA, *g.tmB, g.goff, g.first_group,
        g.ngroups, g.a_rebase, g.out_rebase, g.K, g.n_tiles_n, g.b_rows_per_group, g.epi_mode, g.out, g.ldo, g.err,
        g.res, g.ldr, rp, mblk, g.ksplit > 1 ? g.ksplit : 1, g.partial, g.ldp, g.pstride);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

// K split for launches with few tiles (small batches): the power of two up to
// 8 that fills the persistent CTAs' rounds best (ties to the smaller split),
// keeping at least 8 k-blocks per range.
int grouped_gemm_ksplit(int est_tiles, int nkb, int num_sms) {
    if (est_tiles <= 0) return 1;
    int best = 1;
    double best_eff = 0.0;
    for (int ks = 1; ks <= 8; ks *= 2) {
        if (nkb % ks || nkb / ks < 8) break;
        const long long units = (long long)est_tiles * ks;
        const long long rounds = (units + num_sms - 1) / num_sms;
        const double eff = (double)units / (double)(rounds * num_sms);
        if (eff > best_eff + 1e-9) { best_eff = eff; best = ks; }
    }
    return best;
}

namespace {

// out[row][col] = epilogue(sum over the K ranges, in order, of partial[ks][row][col]).
__global__ void __launch_bounds__(256) splitk_finish_kernel(const int* __restrict__ goff, int first_group,
                                                            int ngroups, int out_rebase, int ksplit,
                                                            const float* __restrict__ partial, int ldp,
                                                            size_t pstride, int epi_mode,
                                                            __nv_bfloat16* __restrict__ out, int ldo) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    const int r0 = out_rebase ? 0 : goff[first_group];
    const int r1 = goff[first_group + ngroups] - (out_rebase ? goff[first_group] : 0);
    const int ncol = epi_mode == EPI_SWIGLU ? ldp / 2 : ldp;
    const long long n = (long long)(r1 - r0) * ncol;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (long long)gridDim.x * blockDim.x) {
        const int r = r0 + (int)(i / ncol);
        const int c = (int)(i % ncol);
        if (epi_mode == EPI_SWIGLU) {
            const int gcol = (c / (BN / 2)) * BN + (c % (BN / 2));
            float gt = 0.f, up = 0.f;
            for (int ks = 0; ks < ksplit; ++ks) {
                const float* pr = partial + (size_t)ks * pstride + (size_t)r * ldp;
                gt += pr[gcol];
                up += pr[gcol + BN / 2];
            }
            out[(size_t)r * ldo + c] = __float2bfloat16_rn(gt / (1.f + __expf(-gt)) * up);
        } else {
            float v = 0.f;
            for (int ks = 0; ks < ksplit; ++ks) v += partial[(size_t)ks * pstride + (size_t)r * ldp + c];
            if (epi_mode == EPI_RELU) v = fmaxf(v, 0.f);
            out[(size_t)r * ldo + c] = __float2bfloat16_rn(v);
        }
    }
}

}  // namespace

cudaError_t launch_splitk_finish(const GemmLaunch& g, int num_sms, cudaStream_t st) {
    if (g.epi_mode != EPI_STORE && g.epi_mode != EPI_SWIGLU && g.epi_mode != EPI_RELU) return cudaErrorInvalidValue;
    const cudaError_t e = launch_pdl(splitk_finish_kernel, dim3(num_sms * 2), dim3(256), 0, st, g.goff, g.first_group,
                                     g.ngroups, g.out_rebase, g.ksplit, g.partial, g.ldp, g.pstride, g.epi_mode, g.out,
                                     g.ldo);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
