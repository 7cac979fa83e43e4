// Kernels (e): the attention sublayer of the full block.
//
// The paper keeps attention on the token's current server and counts it as a
// fixed local term of every layer (Sec. III-C, attention placement); a skip
// bypasses only the FFN sublayer.  The arithmetic is that of the pre-norm
// model families of Sec. VI-A:
//
//   a       = bf16(h * r * gamma_attn),  r = 1/sqrt(mean(h^2) + eps)   (attn_norm_kernel)
//   q, k    = bf16(rope(a W_q^T)), bf16(rope(a W_k^T)), v = bf16(a W_v^T)
//                                  (grouped GEMM, one group, rotary epilogue)
//   o       = softmax(q k^T / sqrt(Dh), causal) v                      (attention_kernel)
//   h_mid   = bf16(h + o W_o^T)                                       (grouped GEMM, residual epilogue)
//
// Tokens are grouped into sequences of S consecutive tokens (one user's
// block); token t sits at position t mod S and attends to positions 0..pos of
// its own sequence.  Every token supplies keys and values (a token that left
// keeps its state, which later tokens still read); outputs of tokens that are
// not live are computed but never read.
//
// The rotary embedding (pairs i, i + Dh/2, angle pos * theta^(-2i/Dh) from a
// host-made cos/sin table) is applied by the projection GEMM's epilogue to the
// fp32 accumulators before their bf16 rounding.
//
// attention_kernel: one CTA per (key/value head, sequence), 320 threads, on
// the 5th-generation tensor cores.  S <= 128 keys fit one tile, so there is no
// running maximum: per query head of the group
//   S = Q K^T          tcgen05.mma M = 128 (queries), N = 128 (keys), K = Dh -> TMEM
//   P = exp(scale (S - max))   causal mask, fp32 (exp as one ex2.approx per
//                      key), rounded to bf16 into shared memory by the 256
//                      softmax threads (two per query row, one per key half;
//                      a warp skips the 32-key chunks above its rows' diagonal)
//   O = P V            tcgen05.mma M = 128, N = Dh, K = 128 keys -> TMEM
//   out = bf16(O / l)  l = the fp32 row sum of the unrounded probabilities
// warp 0 loads K and V of the group once and the query heads one after another
// (TMA, 128-byte swizzle); warp 1 issues the MMAs; warps 2-9 transpose V once
// into a K-major tile (keys contiguous, so that every operand is K-major), then
// run the softmax and the epilogue of each head (two warps per 32 query rows,
// one per half of the keys) while the tensor core computes the next head's
// scores.  Rows past the sequence are loaded (the next
// sequence's rows, or zero fill) but masked as keys and never stored as
// queries.  Every wait is bounded (2 s) and records an error word on expiry.
#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int kSeqMax = 128;

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
    f[0] = bf16_lo(v.x); f[1] = bf16_hi(v.x); f[2] = bf16_lo(v.y); f[3] = bf16_hi(v.y);
    f[4] = bf16_lo(v.z); f[5] = bf16_hi(v.z); f[6] = bf16_lo(v.w); f[7] = bf16_hi(v.w);
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8]) {
    uint4 o;
    o.x = pack_bf16x2(f[0], f[1]);
    o.y = pack_bf16x2(f[2], f[3]);
    o.z = pack_bf16x2(f[4], f[5]);
    o.w = pack_bf16x2(f[6], f[7]);
    return o;
}

// One warp per token row: RMS factor in fp32, then a = bf16(h * r * gamma).
__global__ void __launch_bounds__(256) attn_norm_kernel(const AttnParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    if (blockIdx.x == 0 && threadIdx.x == 0) {
        p.goff[0] = 0;
        p.goff[1] = p.T;
    }
    const int lane = threadIdx.x & 31;
    const int nchunk = p.d >> 3;
    const uint4* gv4 = reinterpret_cast<const uint4*>(p.gamma);
    for (int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; t < p.T; t += (gridDim.x * blockDim.x) >> 5) {
        const uint4* src = reinterpret_cast<const uint4*>(p.h + (size_t)t * p.d);
        float ss = 0.f;
        for (int c = lane; c < nchunk; c += 32) {
            float f[8];
            unpack8(src[c], f);
#pragma unroll
            for (int u = 0; u < 8; ++u) ss = fmaf(f[u], f[u], ss);
        }
        ss = warp_sum_f(ss);
        const float rn = rsqrtf(ss / (float)p.d + p.norm_eps);
        uint4* dst = reinterpret_cast<uint4*>(p.a + (size_t)t * p.d);
        for (int c = lane; c < nchunk; c += 32) {
            float f[8], g[8];
            unpack8(src[c], f);
            unpack8(__ldg(gv4 + c), g);
#pragma unroll
            for (int u = 0; u < 8; ++u) f[u] = f[u] * rn * g[u];
            dst[c] = pack8(f);
        }
    }
}

constexpr int kAttnThreads = 320;            // load warp, MMA warp, 8 softmax / epilogue warps

// Shared-memory layout (byte offsets from a 1024-aligned base).  A box is 128
// rows x 64 bf16 columns (16 KB, 128-byte rows, 128-byte swizzle).
template <int DH>
struct AttnLayout {
    static constexpr int KB = DH / 64;                    // 64-column blocks of a head
    static constexpr int BOX = 128 * 128;
    static constexpr int Q = 0;                           // [KB][128 query rows][128 B]
    static constexpr int K = Q + KB * BOX;                // [KB][128 key rows][128 B]
    static constexpr int V = K + KB * BOX;                // as loaded: [KB][128 key rows][64 dims]
    static constexpr int VT = V + KB * BOX;               // [2 key blocks][DH dim rows][64 keys]
    static constexpr int P = VT + 2 * DH * 128;           // [2 key blocks][128 query rows][64 keys]
    static constexpr int X = P + 2 * BOX;                 // row maxima and sums of the two key halves
    static constexpr int BYTES = X + 4 * 128 * 4;
};

struct __align__(8) AttnBars {
    uint64_t kv, q, vt, s, sfree, pfull, pfree, o, ofree, qfree;
    uint64_t pair[4];          // the two softmax warps of a TMEM lane quarter
    uint32_t tmem_base;
    int abort_flag;
};

template <int DH>
constexpr size_t attn_smem() {
    return 1024 + (size_t)AttnLayout<DH>::BYTES + sizeof(AttnBars);
}

template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 1)
attention_kernel(const __grid_constant__ CUtensorMap tm, const AttnParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    using L = AttnLayout<DH>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t sb = smem_u32(smem);
    AttnBars* bars = reinterpret_cast<AttnBars*>(smem + L::BYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = blockIdx.x, b = blockIdx.y;
    const int G = p.Hq / p.Hkv;                          // query heads per key/value head
    const int t0 = b * p.S;
    const int n = min(p.S, p.T - t0);
    const int kcol = (p.Hq + g) * DH, vcol = (p.Hq + p.Hkv + g) * DH;

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars->kv), 1);
        mbar_init(smem_u32(&bars->q), 1);
        mbar_init(smem_u32(&bars->vt), 8);
        mbar_init(smem_u32(&bars->s), 1);
        mbar_init(smem_u32(&bars->sfree), 8);
        mbar_init(smem_u32(&bars->pfull), 8);
        mbar_init(smem_u32(&bars->pfree), 1);
        mbar_init(smem_u32(&bars->o), 1);
        mbar_init(smem_u32(&bars->ofree), 8);
        for (int j = 0; j < 4; ++j) mbar_init(smem_u32(&bars->pair[j]), 2);
        mbar_init(smem_u32(&bars->qfree), 1);
        bars->abort_flag = 0;
        fence_barrier_init();
        prefetch_tmap(&tm);
    }
    if (warp == 0) tmem_alloc(smem_u32(&bars->tmem_base), 256);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tS = bars->tmem_base, tO = bars->tmem_base + 128;
    volatile int* abort_flag = &bars->abort_flag;

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------- loads
            const uint32_t kvb = smem_u32(&bars->kv);
            mbar_arrive_expect_tx(kvb, 2 * L::KB * L::BOX);
            for (int kb = 0; kb < L::KB; ++kb) {
                tma_load_2d(sb + L::K + kb * L::BOX, &tm, kcol + kb * 64, t0, kvb);
                tma_load_2d(sb + L::V + kb * L::BOX, &tm, vcol + kb * 64, t0, kvb);
            }
            for (int i = 0; i < G; ++i) {
                if (i > 0 && !mbar_wait_bounded(smem_u32(&bars->qfree), (i - 1) & 1, abort_flag, p.err,
                                                ERR_TIMEOUT_ATTN))
                    break;
                const uint32_t qb = smem_u32(&bars->q);
                mbar_arrive_expect_tx(qb, L::KB * L::BOX);
                const int qcol = (g * G + i) * DH;
                for (int kb = 0; kb < L::KB; ++kb) tma_load_2d(sb + L::Q + kb * L::BOX, &tm, qcol + kb * 64, t0, qb);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------------- MMAs
            constexpr uint32_t idS = idesc_bf16_f32(128, 128);
            constexpr uint32_t idO = idesc_bf16_f32(128, DH);
            bool ok = mbar_wait_bounded(smem_u32(&bars->kv), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN) &&
                      mbar_wait_bounded(smem_u32(&bars->vt), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            for (int i = 0; i < G && ok; ++i) {
                const uint32_t ph = i & 1, pph = (i - 1) & 1;
                ok = mbar_wait_bounded(smem_u32(&bars->q), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN) &&
                     (i == 0 || mbar_wait_bounded(smem_u32(&bars->sfree), pph, abort_flag, p.err, ERR_TIMEOUT_ATTN));
                if (!ok) break;
                tc_fence_after();
#pragma unroll
                for (int kb = 0; kb < L::KB; ++kb)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma_bf16(tS, smem_desc_sw128(sb + L::Q + kb * L::BOX + kk * 32),
                                    smem_desc_sw128(sb + L::K + kb * L::BOX + kk * 32), idS, (kb | kk) ? 1u : 0u);
                tc_commit(smem_u32(&bars->s));
                tc_commit(smem_u32(&bars->qfree));
                ok = mbar_wait_bounded(smem_u32(&bars->pfull), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN) &&
                     (i == 0 || mbar_wait_bounded(smem_u32(&bars->ofree), pph, abort_flag, p.err, ERR_TIMEOUT_ATTN));
                if (!ok) break;
                tc_fence_after();
#pragma unroll
                for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma_bf16(tO, smem_desc_sw128(sb + L::P + kb * L::BOX + kk * 32),
                                    smem_desc_sw128(sb + L::VT + kb * DH * 128 + kk * 32), idO, (kb | kk) ? 1u : 0u);
                tc_commit(smem_u32(&bars->o));
                tc_commit(smem_u32(&bars->pfree));
            }
        }
    } else {
        // ----------------------------------------------- softmax and epilogue
        // Eight warps: warps w and w + 4 share TMEM lane quarter qw = w & 3 (32
        // query rows) and take the key halves hk = 0 and 1; a row's maximum
        // and sum combine the halves through shared memory (a two-arrival
        // mbarrier per quarter, bounded waits), and the epilogue splits O's
        // columns the same way.
        const int qw = warp & 3;
        const int hk = (warp - 2) >> 2;
        const int r = qw * 32 + lane;
        const uint32_t loff = (uint32_t)(qw * 32) << 16;
        const int tid = threadIdx.x - 64;              // 0..255
        float* xmax = reinterpret_cast<float*>(smem + L::X);     // [2][128]
        float* xsum = xmax + 256;                                // [2][128]
        const uint32_t pbar = smem_u32(&bars->pair[qw]);
        int ok = 1;
        // Both warps of the pair write, then wait for the pair (phase u of use k).
        auto pair_sync = [&](uint32_t parity) -> int {
            __syncwarp();
            if (lane == 0) mbar_arrive(pbar);
            int w = 1;
            if (lane == 0) w = mbar_wait_bounded(pbar, parity, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            w = __shfl_sync(0xffffffffu, w, 0);
            __syncwarp();
            return w;
        };
        if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->kv), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        if (ok) {
            // V^T: chunk (8 keys) kc of dimension row dim, from V[key][dim].
            for (int idx = tid; idx < DH * 16; idx += 256) {
                const int kc = idx / DH, dim = idx - (idx / DH) * DH;
                const int db = dim >> 6, dc = (dim & 63) >> 3, de = (dim & 7) * 2;
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int k0 = kc * 8 + 2 * e;
                    const uint16_t v0 = *reinterpret_cast<const uint16_t*>(
                        smem + L::V + db * L::BOX + k0 * 128 + ((dc ^ (k0 & 7)) << 4) + de);
                    const uint16_t v1 = *reinterpret_cast<const uint16_t*>(
                        smem + L::V + db * L::BOX + (k0 + 1) * 128 + ((dc ^ ((k0 + 1) & 7)) << 4) + de);
                    w[e] = (uint32_t)v0 | ((uint32_t)v1 << 16);
                }
                *reinterpret_cast<uint4*>(smem + L::VT + (kc >> 3) * DH * 128 + dim * 128 +
                                          (((kc & 7) ^ (dim & 7)) << 4)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->vt));
        }
        const float sl2 = p.scale * 1.4426950408889634f;
        const int kmax = min(r, n - 1);
        // 32-key chunks of this warp's half that some row of the quarter needs.
        const int kq = min(qw * 32 + 31, n - 1);
        for (int i = 0; i < G && ok; ++i) {
            const uint32_t ph = i & 1, pph = (i - 1) & 1;
            if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->s), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            float sv[64];
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                if ((2 * hk + cc) * 32 <= kq) {
                    uint32_t u[32];
                    tmem_ld_32x32(tS + loff + (2 * hk + cc) * 32, u);
                    tmem_ld_wait();
#pragma unroll
                    for (int j = 0; j < 32; ++j) sv[cc * 32 + j] = __uint_as_float(u[j]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->sfree));
            // Causal softmax over keys 0..kmax; exp(x) as 2^(x log2 e), one
            // ex2.approx per key (P is rounded to bf16 next).
            float m = -INFINITY;
#pragma unroll
            for (int cc = 0; cc < 2; ++cc)
                if ((2 * hk + cc) * 32 <= kq)
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (64 * hk + cc * 32 + j <= kmax) m = fmaxf(m, sv[cc * 32 + j]);
            xmax[hk * 128 + r] = m;
            ok = pair_sync(0);
            if (!ok) break;
            m = fmaxf(xmax[r], xmax[128 + r]);
            const float ms = m * sl2;
            float l = 0.f;
#pragma unroll
            for (int cc = 0; cc < 2; ++cc) {
                if ((2 * hk + cc) * 32 <= kq) {
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        float e;
                        asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(fmaf(sv[cc * 32 + j], sl2, -ms)));
                        sv[cc * 32 + j] = (64 * hk + cc * 32 + j <= kmax) ? e : 0.f;
                        l += sv[cc * 32 + j];
                    }
                }
            }
            if (i > 0) {
                if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->pfree), pph, abort_flag, p.err, ERR_TIMEOUT_ATTN);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
            }
#pragma unroll
            for (int c = 0; c < 8; ++c) {
                uint4 w = make_uint4(0u, 0u, 0u, 0u);
                if ((2 * hk + (c >> 2)) * 32 <= kq) {
                    w.x = pack_bf16x2(sv[c * 8 + 0], sv[c * 8 + 1]);
                    w.y = pack_bf16x2(sv[c * 8 + 2], sv[c * 8 + 3]);
                    w.z = pack_bf16x2(sv[c * 8 + 4], sv[c * 8 + 5]);
                    w.w = pack_bf16x2(sv[c * 8 + 6], sv[c * 8 + 7]);
                }
                *reinterpret_cast<uint4*>(smem + L::P + hk * L::BOX + r * 128 + ((c ^ (r & 7)) << 4)) = w;
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->pfull));
            xsum[hk * 128 + r] = l;
            // Epilogue: O / l as bf16, this half's columns, rows of the sequence only.
            if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->o), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            ok = pair_sync(1);
            if (!ok) break;
            tc_fence_after();
            const float il = 1.f / (xsum[r] + xsum[128 + r]);
            __nv_bfloat16* orow = p.out + (size_t)(t0 + min(r, n - 1)) * p.Hq * DH + (size_t)(g * G + i) * DH;
#pragma unroll
            for (int c = hk * (DH / 2); c < (hk + 1) * (DH / 2); c += 32) {
                uint32_t u[32];
                tmem_ld_32x32(tO + loff + c, u);
                tmem_ld_wait();
                if (r < n) {
                    uint4* d4 = reinterpret_cast<uint4*>(orow + c);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(u[8 * q4 + 0]) * il, __uint_as_float(u[8 * q4 + 1]) * il);
                        w.y = pack_bf16x2(__uint_as_float(u[8 * q4 + 2]) * il, __uint_as_float(u[8 * q4 + 3]) * il);
                        w.z = pack_bf16x2(__uint_as_float(u[8 * q4 + 4]) * il, __uint_as_float(u[8 * q4 + 5]) * il);
                        w.w = pack_bf16x2(__uint_as_float(u[8 * q4 + 6]) * il, __uint_as_float(u[8 * q4 + 7]) * il);
                        d4[q4] = w;
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->ofree));
        }
    }
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(bars->tmem_base, 256);
    }
    pdl_trigger();   // the next kernel may be scheduled once every block got here or exited
}

}  // namespace

cudaError_t launch_attn_norm(const AttnParams& p, int num_sms, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    int blocks = (p.T + 7) / 8;
    blocks = blocks < num_sms * 8 ? blocks : num_sms * 8;
    const cudaError_t e = launch_pdl(attn_norm_kernel, dim3(blocks), dim3(256), 0, st, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

cudaError_t launch_attention(const AttnParams& p, const CUtensorMap* tm_qkv, int head_dim, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    if (p.S < 1 || p.S > kSeqMax || p.Hkv < 1 || p.Hq % p.Hkv || !tm_qkv) return cudaErrorInvalidValue;
    static PerDevice attr;
    const cudaError_t ea = (cudaError_t)attr.get([] {
        cudaError_t e = cudaFuncSetAttribute(attention_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)attn_smem<64>());
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(attention_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)attn_smem<128>());
        return (int)e;
    }, true);
    if (ea != cudaSuccess) return ea;
    const dim3 grid(p.Hkv, (p.T + p.S - 1) / p.S);
    cudaError_t e;
    if (head_dim == 64) e = launch_pdl(attention_kernel<64>, grid, dim3(kAttnThreads), attn_smem<64>(), st, *tm_qkv, p);
    else if (head_dim == 128)
        e = launch_pdl(attention_kernel<128>, grid, dim3(kAttnThreads), attn_smem<128>(), st, *tm_qkv, p);
    else return cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
