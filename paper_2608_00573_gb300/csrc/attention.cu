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
// attention_kernel: a unit is one (query head, sequence); persistent CTAs
// (one per SM) take contiguous ranges of units on the 5th-generation tensor
// cores.  S <= 128 keys fit one tile, so there is no running maximum:
//   S = Q K^T   tcgen05.mma M = 128 (queries), N = 128 (keys), K = Dh -> TMEM
//   P = exp(scale (S - max))   causal mask, fp32 (one ex2.approx per key),
//               rounded to bf16 into shared memory over Q, one query row per
//               thread
//   O = P V     tcgen05.mma M = 128, N = Dh, K = 128 keys -> TMEM
//   out = bf16(O / l)   l = the fp32 row sum of the unrounded probabilities
// Two groups of softmax warps take alternate units, and the loads and MMAs of
// the next units run under their softmax and epilogue.
#include <algorithm>

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

constexpr int kAttnThreads = 320;            // load warp, MMA warp, two groups of 4 softmax / epilogue warps
constexpr int kQSlots = 3;                   // Q / P slots in flight
constexpr uint32_t kAttnTmemCols = 512;      // S in two 128-column buffers, O in two DH-column buffers

// Shared-memory layout (byte offsets from a 1024-aligned base).  A box is 128
// rows x 64 bf16 columns (16 KB, 128-byte rows, 128-byte swizzle).  P is
// written over its unit's Q once S = Q K^T has been computed; K and V^T are
// double-buffered per key/value group.
template <int DH>
struct AttnLayout {
    static constexpr int KB = DH / 64;                    // 64-column blocks of a head
    static constexpr int BOX = 128 * 128;
    static constexpr int QP_BYTES = 2 * BOX;              // Q: [KB][128 query rows][128 B]; P: [2][128][128 B]
    static constexpr int K_BYTES = KB * BOX;              // [KB][128 key rows][128 B]
    static constexpr int VT_BYTES = 2 * DH * 128;         // [2 key blocks][DH dim rows][64 keys]
    static constexpr int QP = 0;
    static constexpr int K = QP + kQSlots * QP_BYTES;
    static constexpr int VT = K + 2 * K_BYTES;
    static constexpr int BYTES = VT + 2 * VT_BYTES;
};

struct __align__(8) AttnBars {
    uint64_t q_full[kQSlots], q_empty[kQSlots];
    uint64_t kv_full[2], kv_empty[2];
    uint64_t s_full[2], p_full[2], o_full[2];
    uint32_t tmem_base;
    int abort_flag;
};

template <int DH>
constexpr size_t attn_smem() {
    return 1024 + (size_t)AttnLayout<DH>::BYTES + sizeof(AttnBars);
}

// Units: u = sequence * Hq + query head, so the Hq / Hkv query heads of one
// key/value head and sequence (a group, u / (Hq / Hkv)) are consecutive.
struct AttnUnit {
    int b, hq, g, grp, t0, n;
};

__device__ __forceinline__ AttnUnit attn_unit(const AttnParams& p, int u) {
    AttnUnit a;
    const int R = p.Hq / p.Hkv;
    a.b = u / p.Hq;
    a.hq = u - a.b * p.Hq;
    a.g = a.hq / R;
    a.grp = u / R;
    a.t0 = a.b * p.S;
    a.n = min(p.S, p.T - a.t0);
    return a;
}

// Non-blocking probe of an mbarrier phase (the MMA issuer polls two queues).
__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Persistent: one CTA per SM, each taking a contiguous range of units, so the
// query heads of a group share one load of its K and V^T; 320 threads:
//   warp 0     TMA (one lane): for each new group, K and V^T of the key/value
//              head (rows of the q/k/v projection; the projection's epilogue
//              stores V transposed per sequence, keys contiguous) into the
//              group's buffer (two, alternating); for each unit, Q of its
//              head into the unit's slot (three, in turn); owns the TMEM
//              allocation (512 columns)
//   warp 1     MMAs (one lane), each issued once its inputs are ready:
//              S_i = Q_i K^T (M = 128 queries, N = 128 keys, K = Dh) into S
//              buffer i % 2, and O_i = P_i V (M = 128, N = Dh, K = 128 keys)
//              into O buffer i % 2.  S_i waits until O_{i-2} is issued, that
//              is until the softmax of unit i - 2 has read S buffer i % 2
//   warps 2-9  two groups of four warps, group i % 2 taking unit i, one
//              query row per thread (TMEM lane quarter warp % 4): the row
//              maximum over its causal keys from a first read of S, then
//              p = 2^((s - max) scale log2 e) (one ex2.approx per key; keys
//              past the diagonal or the sequence are 0) from a second read,
//              rounded to bf16 into shared memory over Q, l = the fp32 sum of
//              the unrounded p; finally out = bf16(O / l) for rows of the
//              sequence.  A group starts its next unit only after this
//              epilogue, so its S and O buffers are free by program order.
// Rows past the sequence are loaded (the next sequence's rows, or zero fill)
// and masked as keys, never stored as queries; their V^T slots hold zeros or
// values of an earlier call, which the zero probabilities cancel.  Every wait
// is bounded (2 s) and records an error word on expiry.
template <int DH>
__global__ void __launch_bounds__(kAttnThreads, 1)
attention_kernel(const __grid_constant__ CUtensorMap tm, const __grid_constant__ CUtensorMap tm_vt,
                 const AttnParams p, int nunits) {
    using L = AttnLayout<DH>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    uint8_t* smem = smem_raw + (((raw + 1023u) & ~1023u) - raw);
    const uint32_t sb = smem_u32(smem);
    AttnBars* bars = reinterpret_cast<AttnBars*>(smem + L::BYTES);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int u0 = (int)((long long)blockIdx.x * nunits / gridDim.x);
    const int n = (int)((long long)(blockIdx.x + 1) * nunits / gridDim.x) - u0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kQSlots; ++s) {
            mbar_init(smem_u32(&bars->q_full[s]), 1);
            mbar_init(smem_u32(&bars->q_empty[s]), 1);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bars->kv_full[s]), 1);
            mbar_init(smem_u32(&bars->kv_empty[s]), 1);
            mbar_init(smem_u32(&bars->s_full[s]), 1);
            mbar_init(smem_u32(&bars->p_full[s]), 4);
            mbar_init(smem_u32(&bars->o_full[s]), 1);
        }
        bars->abort_flag = 0;
        fence_barrier_init();
        prefetch_tmap(&tm);
        prefetch_tmap(&tm_vt);
    }
    if (warp == 0) tmem_alloc(smem_u32(&bars->tmem_base), kAttnTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tbase = bars->tmem_base;
    volatile int* abort_flag = &bars->abort_flag;
    pdl_wait();      // q/k/v and V^T written by the projection

    if (warp == 0) {
        if (lane == 0) {
            // ------------------------------------------------------- loads
            int prev = -1, kvn = 0;                      // group of the last unit, groups loaded
            for (int i = 0; i < n && !*abort_flag; ++i) {
                const AttnUnit a = attn_unit(p, u0 + i);
                if (a.grp != prev) {
                    const int ks = kvn & 1;
                    if (kvn >= 2 && !mbar_wait_bounded(smem_u32(&bars->kv_empty[ks]), ((kvn >> 1) - 1) & 1,
                                                       abort_flag, p.err, ERR_TIMEOUT_ATTN))
                        break;
                    const uint32_t fb = smem_u32(&bars->kv_full[ks]);
                    mbar_arrive_expect_tx(fb, L::K_BYTES + L::VT_BYTES);
                    const int kcol = (p.Hq + a.g) * DH;
                    for (int kb = 0; kb < L::KB; ++kb)
                        tma_load_2d(sb + L::K + ks * L::K_BYTES + kb * L::BOX, &tm, kcol + kb * 64, a.t0, fb);
                    const int vrow = (a.b * p.Hkv + a.g) * DH;
                    for (int kb = 0; kb < 2; ++kb)
                        tma_load_2d(sb + L::VT + ks * L::VT_BYTES + kb * DH * 128, &tm_vt, kb * 64, vrow, fb);
                    prev = a.grp;
                    ++kvn;
                }
                const int qs = i % kQSlots, m = i / kQSlots;
                if (m >= 1 && !mbar_wait_bounded(smem_u32(&bars->q_empty[qs]), (m - 1) & 1, abort_flag, p.err,
                                                 ERR_TIMEOUT_ATTN))
                    break;
                const uint32_t qb = smem_u32(&bars->q_full[qs]);
                mbar_arrive_expect_tx(qb, L::KB * L::BOX);
                for (int kb = 0; kb < L::KB; ++kb)
                    tma_load_2d(sb + L::QP + qs * L::QP_BYTES + kb * L::BOX, &tm, a.hq * DH + kb * 64, a.t0, qb);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ------------------------------------------------------- MMAs
            constexpr uint32_t idS = idesc_bf16_f32(128, 128);
            constexpr uint32_t idO = idesc_bf16_f32(128, DH);
            int nS = 0, nO = 0;                          // next unit to get S, O
            int kvc = -1, prevS = -1;                    // ordinal and id of the group of the last S
            int kv_even = 0, kv_odd = 0;                 // K/V buffer of the units between S and O
            bool ok = true;
            uint64_t t_last = globaltimer_ns();
            while (nO < n) {
                bool prog = false;
                if (nS < n && nS <= nO + 1) {
                    const int qs = nS % kQSlots;
                    const int grp = attn_unit(p, u0 + nS).grp;
                    const int kvn = grp != prevS ? kvc + 1 : kvc;
                    if (mbar_test(smem_u32(&bars->q_full[qs]), (nS / kQSlots) & 1) &&
                        (kvn == kvc || mbar_test(smem_u32(&bars->kv_full[kvn & 1]), (kvn >> 1) & 1))) {
                        tc_fence_after();
                        const int ks = kvn & 1;
                        const uint32_t qa = sb + L::QP + qs * L::QP_BYTES, ka = sb + L::K + ks * L::K_BYTES;
                        const uint32_t tS = tbase + (uint32_t)((nS & 1) * 128);
#pragma unroll
                        for (int kb = 0; kb < L::KB; ++kb)
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)
                                tc_mma_bf16(tS, smem_desc_sw128(qa + kb * L::BOX + kk * 32),
                                            smem_desc_sw128(ka + kb * L::BOX + kk * 32), idS, (kb | kk) ? 1u : 0u);
                        tc_commit(smem_u32(&bars->s_full[nS & 1]));
                        if (nS & 1) kv_odd = ks;
                        else kv_even = ks;
                        kvc = kvn;
                        prevS = grp;
                        ++nS;
                        prog = true;
                    }
                }
                if (nO < nS && mbar_test(smem_u32(&bars->p_full[nO & 1]), (nO >> 1) & 1)) {
                    tc_fence_after();
                    const int s = nO & 1, qs = nO % kQSlots, ks = s ? kv_odd : kv_even;
                    const uint32_t pa = sb + L::QP + qs * L::QP_BYTES, va = sb + L::VT + ks * L::VT_BYTES;
                    const uint32_t tO = tbase + 256u + (uint32_t)(s * DH);
#pragma unroll
                    for (int kb = 0; kb < 2; ++kb)
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            tc_mma_bf16(tO, smem_desc_sw128(pa + kb * L::BOX + kk * 32),
                                        smem_desc_sw128(va + kb * DH * 128 + kk * 32), idO, (kb | kk) ? 1u : 0u);
                    tc_commit(smem_u32(&bars->o_full[s]));
                    tc_commit(smem_u32(&bars->q_empty[qs]));
                    if (nO + 1 == n || attn_unit(p, u0 + nO + 1).grp != attn_unit(p, u0 + nO).grp)
                        tc_commit(smem_u32(&bars->kv_empty[ks]));
                    ++nO;
                    prog = true;
                }
                if (prog) {
                    t_last = globaltimer_ns();
                } else {
                    if (*abort_flag) { ok = false; break; }
                    if (globaltimer_ns() - t_last > kTimeoutNs) {
                        *abort_flag = 1;
                        atomicCAS(p.err, 0, ERR_TIMEOUT_ATTN);
                        ok = false;
                        break;
                    }
                }
            }
            // The release commits of the last unit land before the CTA exits.
            if (ok && n > 0) {
                const int last = n - 1;
                if (mbar_wait_bounded(smem_u32(&bars->q_empty[last % kQSlots]), (last / kQSlots) & 1, abort_flag,
                                      p.err, ERR_TIMEOUT_ATTN))
                    mbar_wait_bounded(smem_u32(&bars->kv_empty[kvc & 1]), (kvc >> 1) & 1, abort_flag, p.err,
                                      ERR_TIMEOUT_ATTN);
            }
        }
    } else {
        // ----------------------------------------------- softmax and epilogue
        const int wg = (warp - 2) >> 2;                  // unit parity of this group of warps
        const int qw = warp & 3;                         // TMEM lane quarter of this warp
        const int r = qw * 32 + lane;
        const uint32_t loff = (uint32_t)(qw * 32) << 16;
        const float sl2 = p.scale * 1.4426950408889634f;
        for (int i = wg; i < n; i += 2) {
            const AttnUnit a = attn_unit(p, u0 + i);
            const int qs = i % kQSlots;
            const uint32_t ph = (uint32_t)(i >> 1) & 1u;
            const int kmax = min(r, a.n - 1);            // causal keys of this row
            const int kq = min(qw * 32 + 31, a.n - 1);   // largest key any row of the quarter needs
            const uint32_t tS = tbase + loff + (uint32_t)(wg * 128);
            const uint32_t tO = tbase + loff + 256u + (uint32_t)(wg * DH);
            uint8_t* sP = smem + L::QP + qs * L::QP_BYTES;
            int ok = 1;
            if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->s_full[wg]), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            float m = -INFINITY;
#pragma unroll 1
            for (int cc = 0; cc < 4; ++cc) {
                if (cc * 32 > kq) break;
                uint32_t u[32];
                tmem_ld_32x32(tS + cc * 32, u);
                tmem_ld_wait();
#pragma unroll
                for (int j = 0; j < 32; ++j)
                    if (cc * 32 + j <= kmax) m = fmaxf(m, __uint_as_float(u[j]));
            }
            const float ms = m * sl2;
            float l = 0.f;
#pragma unroll 1
            for (int cc = 0; cc < 4; ++cc) {
                uint4 w[4];
                if (cc * 32 <= kq) {
                    uint32_t u[32];
                    tmem_ld_32x32(tS + cc * 32, u);
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
                    *reinterpret_cast<uint4*>(sP + (cc >> 1) * L::BOX + r * 128 + ((c16 ^ (r & 7)) << 4)) = w[q4];
                }
            }
            tc_fence_before();
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bars->p_full[wg]));
            if (lane == 0) ok = mbar_wait_bounded(smem_u32(&bars->o_full[wg]), ph, abort_flag, p.err, ERR_TIMEOUT_ATTN);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            // Epilogue: out = bf16(O / l), rows of the sequence only.
            tc_fence_after();
            const float il = 1.f / l;
            __nv_bfloat16* orow = p.out + (size_t)(a.t0 + min(r, a.n - 1)) * p.Hq * DH + (size_t)a.hq * DH;
#pragma unroll 1
            for (int c = 0; c < DH; c += 32) {
                uint32_t u[32];
                tmem_ld_32x32(tO + c, u);
                tmem_ld_wait();
                if (r < a.n) {
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
            tc_fence_before();
        }
    }
    __syncthreads();
    if (warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tbase, kAttnTmemCols);
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
                             int num_sms, cudaStream_t st) {
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
    // One persistent CTA per SM (at most one per unit), units split evenly.
    const long long units = (long long)p.Hq * ((p.T + p.S - 1) / p.S);
    if (units > (1LL << 30)) return cudaErrorInvalidValue;
    const dim3 grid((unsigned)std::min<long long>(units, num_sms));
    cudaError_t e;
    if (head_dim == 64)
        e = launch_pdl(attention_kernel<64>, grid, dim3(kAttnThreads), attn_smem<64>(), st, *tm_qkv, *tm_vt, p,
                       (int)units);
    else if (head_dim == 128)
        e = launch_pdl(attention_kernel<128>, grid, dim3(kAttnThreads), attn_smem<128>(), st, *tm_qkv, *tm_vt, p,
                       (int)units);
    else return cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
