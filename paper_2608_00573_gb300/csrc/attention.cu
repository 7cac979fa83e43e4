// Kernels (e): the attention sublayer of the full block.
//
// The paper keeps attention on the token's current server and counts it as a
// fixed local term of every layer (Sec. III-C, attention placement); a skip
// bypasses only the FFN sublayer.  The arithmetic is that of the pre-norm
// model families of Sec. VI-A:
//
//   a       = bf16(h * r * gamma_attn),  r = 1/sqrt(mean(h^2) + eps)   (attn_norm_kernel)
//   q, k    = bf16(rope(a W_q^T)), bf16(rope(a W_k^T)), v = bf16(a W_v^T)
//                                  (grouped GEMM, one group, rotary epilogue;
//                                  v is stored transposed per sequence)
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
// fp32 accumulators before their bf16 rounding.  The same epilogue writes the
// value heads as V^T[sequence][value dim][key slot] (128 slots per sequence),
// the K-major operand of O = P V.
//
// attention_kernel: one CTA per (query head, sequence), 192 threads, two
// CTAs per SM (three at head_dim 64), on the 5th-generation tensor cores.
// S <= 128 keys fit one tile, so there is no running maximum:
//   S = Q K^T   tcgen05.mma M = 128 (queries), N = 128 (keys), K = Dh -> TMEM
//   P = exp(scale (S - max))   causal mask, fp32 (one ex2.approx per key),
//               rounded to bf16 into shared memory over Q by four warps, one
//               query row per thread
//   O = P V     tcgen05.mma M = 128, N = Dh, K = 128 keys -> the same TMEM columns
//   out = bf16(O / l)   l = the fp32 row sum of the unrounded probabilities
// Several CTAs per SM overlap one CTA's loads with another's softmax.
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

constexpr int kAttnThreads = 192;            // load warp, MMA warp, 4 softmax / epilogue warps

// Shared-memory layout (byte offsets from a 1024-aligned base).  A box is 128
// rows x 64 bf16 columns (16 KB, 128-byte rows, 128-byte swizzle).  P is
// written over Q once S = Q K^T has been computed.
template <int DH>
struct AttnLayout {
    static constexpr int KB = DH / 64;                    // 64-column blocks of a head
    static constexpr int BOX = 128 * 128;
    static constexpr int QP = 0;                          // Q: [KB][128 query rows][128 B]; P: [2][128][128 B]
    static constexpr int K = QP + 2 * BOX;                // [KB][128 key rows][128 B]
    static constexpr int VT = K + KB * BOX;               // [2 key blocks][DH dim rows][64 keys]
    static constexpr int BYTES = VT + 2 * DH * 128;
};

struct __align__(8) AttnBars {
    uint64_t ldqk, ldv, s, p, o;
    uint32_t tmem_base;
    int abort_flag;
};

template <int DH>
constexpr size_t attn_smem() {
    return 1024 + (size_t)AttnLayout<DH>::BYTES + sizeof(AttnBars);
}

// One CTA per (query head, sequence), 192 threads, two or three CTAs per SM:
//   warp 0     TMA: Q of the head, K of its key/value head (rows of the q/k/v
//              projection) and V^T of the key/value head (the projection's
//              epilogue stores V transposed per sequence, keys contiguous);
//              owns the TMEM allocation (128 columns)
//   warp 1     S = Q K^T (M = 128 queries, N = 128 keys, K = Dh) into TMEM,
//              then O = P V (M = 128, N = Dh, K = 128 keys) into the same
//              columns once every row of S has been read
//   warps 2-5  one query row per thread (TMEM lane quarter warp % 4): the row
//              maximum over its causal keys from a first read of S, then
//              p = 2^((s - max) scale log2 e) (one ex2.approx per key; keys
//              past the diagonal or the sequence are 0) from a second read,
//              rounded to bf16 into shared memory over Q, l = the fp32 sum of
//              the unrounded p; finally out = bf16(O / l) for rows of the
//              sequence
// Rows past the sequence are loaded (the next sequence's rows, or zero fill)
// and masked as keys, never stored as queries; their V^T slots hold zeros or
// values of an earlier call, which the zero probabilities cancel.  Every wait
// is bounded (2 s) and records an error word on expiry.
template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 2)
attention_kernel(const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tm_vt,
                 const AttnParams p) {
    using L = AttnLayout<DH>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t sb = smem_u32(smem);
    AttnBars* bars = reinterpret_cast<AttnBars*>(smem + L::BYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int hq = blockIdx.x, b = blockIdx.y;
    const int g = hq / (p.Hq / p.Hkv);                   // key/value head of this query head
    const int t0 = b * p.S;
    const int n = min(p.S, p.T - t0);

    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bars->ldqk), 1);
        mbar_init(smem_u32(&bars->ldv), 1);
        mbar_init(smem_u32(&bars->s), 1);
        mbar_init(smem_u32(&bars->p), 4);
        mbar_init(smem_u32(&bars->o), 1);
        bars->abort_flag = 0;
        fence_barrier_init();
        prefetch_tmap(&tm);
        prefetch_tmap(&tm_vt);
    }
    if (warp == 0) tmem_alloc(smem_u32(&bars->tmem_base), 128);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tS = bars->tmem_base;                 // S, then O in the same columns
    volatile int* abort_flag = &bars->abort_flag;
    pdl_wait();      // q/k/v and V^T written by the projection

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------- loads
            // Q and K first (S needs them), V^T behind them (only O needs it).
            const uint32_t lb = smem_u32(&bars->ldqk), vb = smem_u32(&bars->ldv);
            mbar_arrive_expect_tx(lb, 2 * L::KB * L::BOX);
            const int qcol = hq * DH, kcol = (p.Hq + g) * DH;
            for (int kb = 0; kb < L::KB; ++kb) {
                tma_load_2d(sb + L::QP + kb * L::BOX, &tm, qcol + kb * 64, t0, lb);
                tma_load_2d(sb + L::K + kb * L::BOX, &tm, kcol + kb * 64, t0, lb);
            }
            mbar_arrive_expect_tx(vb, 2 * DH * 128);
            const int vrow = (b * p.Hkv + g) * DH;
            for (int kb = 0; kb < 2; ++kb) tma_load_2d(sb + L::VT + kb * DH * 128, &tm_vt, kb * 64, vrow, vb);
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------------- MMAs
            constexpr uint32_t idS = idesc_bf16_f32(128, 128);
            constexpr uint32_t idO = idesc_bf16_f32(128, DH);
            if (mbar_wait_bounded(smem_u32(&bars->ldqk), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN)) {
                tc_fence_after();
#pragma unroll
                for (int kb = 0; kb < L::KB; ++kb)
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)
                        tc_mma_bf16(tS, smem_desc_sw128(sb + L::QP + kb * L::BOX + kk * 32),
                                    smem_desc_sw128(sb + L::K + kb * L::BOX + kk * 32), idS, (kb | kk) ? 1u : 0u);
                tc_commit(smem_u32(&bars->s));
                if (mbar_wait_bounded(smem_u32(&bars->p), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN) &&
                    mbar_wait_bounded(smem_u32(&bars->ldv), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN)) {
                    tc_fence_after();
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc_mma_bf16(tS, smem_desc_sw128(sb + L::QP + kb * L::BOX + kk * 32),
                                        smem_desc_sw128(sb + L::VT + kb * DH * 128 + kk * 32), idO,
                                        (kb | kk) ? 1u : 0u);
                    tc_commit(smem_u32(&bars->o));
                }
            }
        }
    } else {
        // ----------------------------------------------- softmax and epilogue
        const int qw = warp & 3;                         // TMEM lane quarter of this warp
        const int r = qw * 32 + lane;
        const uint32_t loff = (uint32_t)(qw * 32) << 16;
        const int kmax = min(r, n - 1);                  // causal keys of this row
        const int kq = min(qw * 32 + 31, n - 1);         // largest key any row of the quarter needs
        const float sl2 = p.scale * 1.4426950408889634f;
        int ok = 1;
        if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->s), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN);
        ok = __shfl_sync(0xffffffffu, ok, 0);
        float l = 0.f;
        if (ok) {
            tc_fence_after();
            float m = -INFINITY;
#pragma unroll 1
            for (int cc = 0; cc < 4; ++cc) {
                if (cc * 32 > kq) break;
                uint32_t u[32];
                tmem_ld_32x32(tS + loff + cc * 32, u);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (cc * 32 + j <= kmax) m = fmaxf(m, __uint_as_float(u[j]));
            }
            const float ms = m * sl2;
#pragma unroll 1
            for (int cc = 0; cc < 4; ++cc) {
                uint4 w[4];
                if (cc * 32 <= kq) {
                    uint32_t u[32];
                    tmem_ld_32x32(tS + loff + cc * 32, u);
                    tmem_ld_wait();
                    float e[32];
#pragma unroll
                    for (int j = 0; j < 32; ++j) {
                        float x;
                        asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(x) : "f"(fmaf(__uint_as_float(u[j]), sl2, -ms)));
                        e[j] = (cc * 32 + j <= kmax) ? x : 0.f;
                        l += e[j];
                    }
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4)
                        w[q4] = make_uint4(pack_bf16x2(e[8 * q4 + 0], e[8 * q4 + 1]),
                                           pack_bf16x2(e[8 * q4 + 2], e[8 * q4 + 3]),
                                           pack_bf16x2(e[8 * q4 + 4], e[8 * q4 + 5]),
                                           pack_bf16x2(e[8 * q4 + 6], e[8 * q4 + 7]));
                } else {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) w[q4] = make_uint4(0u, 0u, 0u, 0u);
                }
                // keys [32 cc, 32 cc + 32): key block cc / 2, 16-byte chunks (cc & 1) * 4 + q4
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const int c16 = (cc & 1) * 4 + q4;
                    *reinterpret_cast<uint4*>(smem + L::QP + (cc >> 1) * L::BOX + r * 128 + ((c16 ^ (r & 7)) << 4)) =
                        w[q4];
                }
            }
            tc_fence_before();
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->p));
            if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->o), 0, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            ok = __shfl_sync(0xffffffffu, ok, 0);
        }
        if (ok) {
            // Epilogue: out = bf16(O / l), rows of the sequence only.
            tc_fence_after();
            const float il = 1.f / l;
            __nv_bfloat16* orow = p.out + (size_t)(t0 + min(r, n - 1)) * p.Hq * DH + (size_t)hq * DH;
#pragma unroll 1
            for (int c = 0; c < DH; c += 32) {
                uint32_t u[32];
                tmem_ld_32x32(tS + loff + c, u);
                tmem_ld_wait();
                if (r < n) {
                    uint4* d4 = reinterpret_cast<uint4*>(orow + c);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4)
                        d4[q4] = make_uint4(pack_bf16x2(__uint_as_float(u[8 * q4 + 0]) * il,
                                                        __uint_as_float(u[8 * q4 + 1]) * il),
                                            pack_bf16x2(__uint_as_float(u[8 * q4 + 2]) * il,
                                                        __uint_as_float(u[8 * q4 + 3]) * il),
                                            pack_bf16x2(__uint_as_float(u[8 * q4 + 4]) * il,
                                                        __uint_as_float(u[8 * q4 + 5]) * il),
                                            pack_bf16x2(__uint_as_float(u[8 * q4 + 6]) * il,
                                                        __uint_as_float(u[8 * q4 + 7]) * il));
                }
            }
        }
        tc_fence_before();
    }
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(bars->tmem_base, 128);
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

cudaError_t launch_attention(const AttnParams& p, const CUtensorMap* tm_qkv, const CUtensorMap* tm_vt, int head_dim,
                             cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    if (p.S < 1 || p.S > kSeqMax || p.Hkv < 1 || p.Hq % p.Hkv || !tm_qkv || !tm_vt) return cudaErrorInvalidValue;
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
    const dim3 grid(p.Hq, (p.T + p.S - 1) / p.S);
    cudaError_t e;
    if (head_dim == 64)
        e = launch_pdl(attention_kernel<64>, grid, dim3(kAttnThreads), attn_smem<64>(), st, *tm_qkv, *tm_vt, p);
    else if (head_dim == 128)
        e = launch_pdl(attention_kernel<128>, grid, dim3(kAttnThreads), attn_smem<128>(), st, *tm_qkv, *tm_vt, p);
    else return cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
