// Kernel (a0): router and exit-head dot products of a layer on the tensor cores.
//
//   z[t][e]     = r_t * sum_i h[t][i] * gamma_i * W_r[e][i] + b_r[e]     e < E   (Eq. 4 input)
//   z[t][E + c] = r_t * sum_i h[t][i] * W_x[c][i]            + b_x[c]     c < C   (Eq. 7 input)
// with r_t = 1/sqrt(mean_i h[t][i]^2 + eps) (1 without the pre-FFN RMSNorm).
// The columns i are split into ksplit ranges; each (128-token tile, column
// range) unit writes its partial sums (and partial sums of h^2; a token's
// ranges are contiguous: [T][ksplit][zs]), and the
// decision kernel adds the ranges in a fixed order before applying r and the
// bias.
//
// The router's gamma * W_r products are exact in fp32 and split exactly into
// two bf16 matrices (hi + lo), so two bf16 MMAs give the logits without
// rounding the normalised input.  Each 64-column slab starts its MMAs from
// zero and the slab's sums are added to IEEE fp32 registers (__fadd_rn): the
// tensor core's own accumulation then only touches sums of 64 (hi) + 64 (lo)
// exact products, which keeps the logits at fp32 accuracy (the decisions
// compare them to 1e-5).  The sum of squares comes from the same fragments:
// two more MMAs per 16-column step multiply the 16-token A fragment by itself
// (its rows reused as the B operand), and the diagonal of the resulting 16 x 16
// Gram block is each token's partial sum of h^2.
//
// Design (persistent, 288 threads per CTA, two CTAs per SM):
//   warp 8      producer (one lane): per 64-column slab, 2-D TMA boxes of the
//               128-token hidden tile and of the pass's weight rows (hi and
//               lo), 128-byte swizzle, rows past the tensor zero-filled, into a
//               ring of up to 8 stages guarded by full/empty mbarriers
//   warps 0-7   16 tokens each: ldmatrix + mma.sync m16n8k16 (bf16 in, fp32
//               accumulate), up to 32 output rows per pass over h
// Hidden rows of dead tokens are loaded with their tile but never stored.
// Every wait is bounded (2 s); on expiry the kernel records an error word and
// returns.
#include <algorithm>

#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int kTok = 128;         // tokens per tile (8 consumer warps x 16)
constexpr int kKS = 64;           // columns per slab (one 128-byte row per token / weight)
constexpr int kNG = 32;           // largest number of outputs per pass (4 n-tiles of 8)
constexpr int kConsumers = kTok / 16;
constexpr int kThreads = 32 * (kConsumers + 1);
constexpr int kA = kTok * kKS * 2;     // 16 KB hidden slab, 128-byte swizzled
constexpr int kMaxStages = 8;

struct __align__(8) RouterBars {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    int abort_flag;
};

// Stage: hidden slab, then ng weight rows (hi), then nl (lo), all dense
// 128-byte rows with 128-byte swizzle (1024-byte aligned, ng and nl % 8 == 0).
__host__ __device__ __forceinline__ size_t stage_bytes(int ng, int nl) {
    return (size_t)kA + (size_t)(ng + nl) * kKS * 2;
}

// Shared memory per CTA: two CTAs per SM.
constexpr size_t kSmemBudget = 100 * 1024;

int stages_for(int ng, int nl) {
    const size_t sb = stage_bytes(ng, nl);
    const int s = (int)((kSmemBudget - 1024 - sizeof(RouterBars)) / sb);
    return std::max(2, std::min(kMaxStages, s));
}

size_t smem_for(int ng, int nl, int stages) {
    return 1024 + (size_t)stages * stage_bytes(ng, nl) + sizeof(RouterBars);
}

// Address of 16-byte chunk c of row r in a 128-byte-swizzled tile.
__device__ __forceinline__ uint32_t sw128(uint32_t base, int r, int c) {
    return base + (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4));
}

// NT: n-tiles of 8 outputs per pass (ng = 8 NT rows, the last ones past n_out
// zero-filled by TMA and never stored): 1, 2 or 4.
template <int NT>
__global__ void __launch_bounds__(kThreads, 2)
router_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmBhi,
              const __grid_constant__ CUtensorMap tmBlo, const RouterParams p, int stages) {
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const int NG = p.ng, NL = p.nl;
    const size_t sbytes = stage_bytes(NG, NL);
    RouterBars* bars = reinterpret_cast<RouterBars*>(smem + (size_t)stages * sbytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const int nslab = p.d / kKS / p.ksplit;
    const int ntile = (p.T + kTok - 1) / kTok;
    const int npass = (p.n_out + NG - 1) / NG;
    const int nunits = ntile * p.ksplit * npass;   // unit u: pass u / (ntile*ksplit), then tile, then range

    if (threadIdx.x == 0) {
        for (int s = 0; s < stages; ++s) {
            mbar_init(smem_u32(&bars->full[s]), 1);
            mbar_init(smem_u32(&bars->empty[s]), kConsumers);
        }
        bars->abort_flag = 0;
        fence_barrier_init();
        prefetch_tmap(&tmA);
        prefetch_tmap(&tmBhi);
        if (NL > 0) prefetch_tmap(&tmBlo);
    }
    __syncthreads();
    pdl_wait();      // hidden states and liveness written by the preceding kernels
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    volatile int* abort_flag = &bars->abort_flag;

    if (warp == kConsumers) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int it = 0;
            for (int u = blockIdx.x; u < nunits && !*abort_flag; u += gridDim.x) {
                const int pass = u / (ntile * p.ksplit);
                const int rem = u - pass * ntile * p.ksplit;
                const int tile = rem / p.ksplit;
                const int kr = rem - tile * p.ksplit;
                const int ng0 = pass * NG;
                const bool lo = ng0 < p.n_lo && NL > 0;
                const uint32_t tx = (uint32_t)kA + (uint32_t)(NG + (lo ? NL : 0)) * (kKS * 2);
                bool ok = true;
                for (int sl = 0; sl < nslab; ++sl, ++it) {
                    const int s = it % stages;
                    const uint32_t ph = (it / stages) & 1;
                    if (!mbar_wait_bounded(smem_u32(&bars->empty[s]), ph ^ 1, abort_flag, p.err, ERR_TIMEOUT_ROUTER)) {
                        ok = false;
                        break;
                    }
                    const int col = (kr * nslab + sl) * kKS;
                    const uint32_t fb = smem_u32(&bars->full[s]);
                    const uint32_t st0 = smem_u32(smem + (size_t)s * sbytes);
                    mbar_arrive_expect_tx(fb, tx);
                    tma_load_2d(st0, &tmA, col, tile * kTok, fb);
                    tma_load_2d(st0 + kA, &tmBhi, col, ng0, fb);
                    if (lo) tma_load_2d(st0 + kA + NG * kKS * 2, &tmBlo, col, ng0, fb);
                }
                if (!ok) break;
            }
        }
    } else {
        // ------------------------------------------------------------ consumers
        const int g = lane >> 2, tig = lane & 3;
        // Lane (g, g / 2) holds tokens g and 8 + g of the Gram diagonal.
        const bool diag = (tig == (g >> 1));
        const int dq = g & 1;
        // Per-lane ldmatrix offsets in the 128-byte-swizzled tiles, one per k step.
        const int ar = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
        const int br = lane & 7;
        uint32_t a_off[kKS / 16], b_off[kKS / 16];
#pragma unroll
        for (int kk = 0; kk < kKS / 16; ++kk) {
            a_off[kk] = (uint32_t)(ar * 128 + (((kk * 2 + (lane >> 4)) ^ (ar & 7)) << 4));
            b_off[kk] = (uint32_t)(br * 128 + (((kk * 2 + ((lane >> 3) & 1)) ^ br) << 4));
        }
        const int nlt = NL / 8;                 // n-tiles with a lo part in a pass
        int it = 0;
        for (int u = blockIdx.x; u < nunits; u += gridDim.x) {
            const int pass = u / (ntile * p.ksplit);
            const int rem = u - pass * ntile * p.ksplit;
            const int tile = rem / p.ksplit;
            const int kr = rem - tile * p.ksplit;
            const int ng0 = pass * NG;
            const int nrows = min(NG, p.n_out - ng0);
            const int lo_t = ng0 < p.n_lo ? min(nlt, (p.n_lo - ng0 + 7) / 8) : 0;
            float acc[NT][4];
#pragma unroll
            for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
            float sq0 = 0.f, sq1 = 0.f;
            // Liveness of this lane's two output rows, loaded now so that the
            // stores after the last slab do not wait on it.
            const int t_lo = tile * kTok + warp * 16 + g, t_hi = t_lo + 8;
            const bool st_lo = t_lo < p.T && p.alive[t_lo];
            const bool st_hi = t_hi < p.T && p.alive[t_hi];
            bool ok = true;
            for (int sl = 0; sl < nslab; ++sl, ++it) {
                const int s = it % stages;
                const uint32_t ph = (it / stages) & 1;
                int w = 1;
                if (lane == 0) w = mbar_wait_bounded(smem_u32(&bars->full[s]), ph, abort_flag, p.err, ERR_TIMEOUT_ROUTER);
                w = __shfl_sync(0xffffffffu, w, 0);
                if (!w) { ok = false; break; }
                const uint32_t sA = smem_u32(smem + (size_t)s * sbytes);
                const uint32_t sBh = sA + kA;
                const uint32_t sBl = sBh + NG * kKS * 2;
                // One slab: the tensor core sums its 64 (hi) + 64 (lo) exact
                // products per output; the slab sums are then added in IEEE fp32.
                float part[NT][4];
#pragma unroll
                for (int j = 0; j < NT; ++j) part[j][0] = part[j][1] = part[j][2] = part[j][3] = 0.f;
                float g0[4] = {0.f, 0.f, 0.f, 0.f}, g1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int kk = 0; kk < kKS / 16; ++kk) {
                    uint32_t a[4];
                    ldmatrix_x4(a, sA + a_off[kk]);
#pragma unroll
                    for (int j = 0; j < NT; ++j) {
                        uint32_t b[2];
                        ldmatrix_x2(b, sBh + j * 1024 + b_off[kk]);
                        mma_bf16_16816(part[j], a, b);
                        if (j < lo_t) {
                            ldmatrix_x2(b, sBl + j * 1024 + b_off[kk]);
                            mma_bf16_16816(part[j], a, b);
                        }
                    }
                    if (pass == 0) {
                        // Gram blocks: tokens 0-7 and 8-15 of the fragment as B.
                        const uint32_t b0[2] = {a[0], a[2]}, b1[2] = {a[1], a[3]};
                        mma_bf16_16816(g0, a, b0);
                        mma_bf16_16816(g1, a, b1);
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_u32(&bars->empty[s]));
#pragma unroll
                for (int j = 0; j < NT; ++j)
#pragma unroll
                    for (int q = 0; q < 4; ++q) acc[j][q] = __fadd_rn(acc[j][q], part[j][q]);
                sq0 = __fadd_rn(sq0, dq ? g0[1] : g0[0]);
                sq1 = __fadd_rn(sq1, dq ? g1[3] : g1[2]);
            }
            if (!ok) break;
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const int t = half ? t_hi : t_lo;
                if (!(half ? st_hi : st_lo)) continue;
                if (pass == 0 && diag) p.sqpart[(size_t)t * p.ksplit + kr] = half ? sq1 : sq0;
                float* zrow = p.zpart + ((size_t)t * p.ksplit + kr) * p.zs;
#pragma unroll
                for (int j = 0; j < NT; ++j) {
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        const int col = j * 8 + tig * 2 + q;
                        if (col < nrows) zrow[ng0 + col] = acc[j][half * 2 + q];
                    }
                }
            }
        }
    }
}

}  // namespace

int router_lo_rows(int n_lo, int ng) {
    const int r = ((n_lo + 7) / 8) * 8;
    return r < ng ? r : ng;
}

// Rows per pass: n-tiles of 8 rounded up to 1, 2 or 4 (the kernel's register
// tile), at most 32: wider passes need the registers of a whole SM per CTA,
// and a second CTA per SM (plus a re-read of h per extra pass) was faster.
int router_pass_rows(int n_out) {
    const int t = (n_out + 7) / 8;
    const int nt = t <= 1 ? 1 : t <= 2 ? 2 : 4;
    return nt * 8;
}

// Column ranges per launch: the smallest power of two dividing d/64 that gives
// every SM at least one (tile, range, pass) unit, and at most kMaxSplit.  More
// ranges only add partial sums for the decision kernel to write and read
// back: on the 8192-token layer with d = 2048 and 60 experts, 2 ranges took
// 27 us where 32 ranges (eight units per SM) took 50 us; and for a
// decode-sized batch (one 128-token tile) the decision kernel's per-token
// sums over 64 ranges cost more than the router saves with them.
constexpr int kMaxSplit = 16;

int router_ksplit(int T, int d, int n_out, int num_sms) {
    const int nslab = d / kKS;
    const int tiles = (T + kTok - 1) / kTok;
    const int ng = router_pass_rows(n_out);
    const long long units = (long long)tiles * ((n_out + ng - 1) / ng);
    int ks = 1;
    while (ks < nslab && ks < kMaxSplit && units * ks < num_sms && nslab % (ks * 2) == 0) ks *= 2;
    return ks;
}

cudaError_t launch_router(const CUtensorMap* tmA, const CUtensorMap* tmBhi, const CUtensorMap* tmBlo,
                          const RouterParams& p, int num_sms, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    if (p.d % kKS || p.ksplit < 1 || (p.d / kKS) % p.ksplit || p.ng < 8 || p.ng > kNG || p.ng % 8 ||
        p.nl < 0 || p.nl > p.ng || p.nl % 8 || !tmA || !tmBhi || (p.nl > 0 && !tmBlo))
        return cudaErrorInvalidValue;
    static PerDevice attr;
    const cudaError_t ea = (cudaError_t)attr.get([] {
        cudaError_t e = cudaSuccess;
        for (const void* f : {(const void*)router_kernel<1>, (const void*)router_kernel<2>, (const void*)router_kernel<4>})
            if (e == cudaSuccess) e = cudaFuncSetAttribute(f, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kSmemBudget);
        return (int)e;
    }, true);
    if (ea != cudaSuccess) return ea;
    const int nt = p.ng / 8;
    if (nt != 1 && nt != 2 && nt != 4) return cudaErrorInvalidValue;
    const int stages = stages_for(p.ng, p.nl);
    const size_t smem = smem_for(p.ng, p.nl, stages);
    const int ntile = (p.T + kTok - 1) / kTok;
    const int npass = (p.n_out + p.ng - 1) / p.ng;
    const long long units = (long long)ntile * p.ksplit * npass;
    const int grid = (int)std::min<long long>(units, 2LL * num_sms);
    const CUtensorMap* lo = p.nl > 0 ? tmBlo : tmBhi;
    cudaError_t e;
    if (nt == 1) e = launch_pdl(router_kernel<1>, dim3(grid), dim3(kThreads), smem, st, *tmA, *tmBhi, *lo, p, stages);
    else if (nt == 2) e = launch_pdl(router_kernel<2>, dim3(grid), dim3(kThreads), smem, st, *tmA, *tmBhi, *lo, p, stages);
    else e = launch_pdl(router_kernel<4>, dim3(grid), dim3(kThreads), smem, st, *tmA, *tmBhi, *lo, p, stages);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
