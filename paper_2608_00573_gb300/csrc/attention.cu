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
// attention_kernel: one block per (query head, sequence), 4 warps.  Q, K and V
// of the sequence (S <= 128 rows) are staged in padded shared memory by
// cp.async with every load in flight at once.  Each warp owns two 16-row query blocks
// (mb and 7 - mb, which balances the causal work), computes the full causal
// score rows with mma.sync m16n8k16 (bf16 in, fp32 accumulate), takes the
// softmax in fp32 registers (quad shuffles), rounds the probabilities to bf16
// as the A operand of the P.V product (V fragments by ldmatrix.trans), divides
// by the fp32 row sums and writes bf16 rows through shared memory with 16-byte
// stores.  The contraction is small (S x S x Dh per head) next to the
// projections, so the legacy mma.sync path is used; the projections are the
// tcgen05 grouped GEMM.
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

template <int DH>
__global__ void __launch_bounds__(128) attention_kernel(const AttnParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    constexpr int LD = DH + 8;                 // padded row (bf16): conflict-free ldmatrix
    constexpr int NTO = DH / 8;                // output n-tiles
    extern __shared__ __align__(16) uint8_t sm[];
    __nv_bfloat16* sQ = reinterpret_cast<__nv_bfloat16*>(sm);
    __nv_bfloat16* sK = sQ + kSeqMax * LD;
    __nv_bfloat16* sV = sK + kSeqMax * LD;

    const int hq = blockIdx.x, b = blockIdx.y;
    const int g = hq / (p.Hq / p.Hkv);
    const int t0 = b * p.S;
    const int n = min(p.S, p.T - t0);
    const int n16 = (n + 15) & ~15;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const size_t qoff = (size_t)hq * DH;
    const size_t koff = (size_t)(p.Hq + g) * DH;
    const size_t voff = (size_t)(p.Hq + p.Hkv + g) * DH;

    // Stage Q, K and V of the sequence (the projection's epilogue has already
    // rotated Q and K) with every load in flight at once; rows >= n are zero.
    constexpr int RC = DH / 8;                 // 16-byte chunks per row
    for (int i = tid; i < 3 * n16 * RC; i += 128) {
        const int which = i / (n16 * RC);      // 0: query head, 1: key head, 2: value head
        const int rem = i - which * n16 * RC;
        const int r = rem / RC, c = (rem - r * RC) * 8;
        __nv_bfloat16* dst = (which == 0 ? sQ : which == 1 ? sK : sV) + r * LD + c;
        const size_t off = which == 0 ? qoff : which == 1 ? koff : voff;
        const bool ok = r < n;
        const __nv_bfloat16* src = p.qkv + (size_t)(t0 + (ok ? r : 0)) * p.nqkv + off + c;
        cp_async16(smem_u32(dst), src, ok ? 16 : 0);
    }
    cp_async_commit();
    cp_async_wait<0>();
    __syncthreads();

    const int gq = lane >> 2, tig = lane & 3;
    const int nmb = n16 >> 4;
    const size_t ostride = (size_t)p.Hq * DH;
#pragma unroll 1
    for (int pass = 0; pass < 2; ++pass) {
        const int mb = pass == 0 ? warp : 7 - warp;
        if (mb >= nmb) continue;
        const int nt = 2 * (mb + 1);            // key tiles of 8 up to the block's last row
        float s[16][4];
#pragma unroll
        for (int j = 0; j < 16; ++j) s[j][0] = s[j][1] = s[j][2] = s[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < DH / 16; ++kk) {
            uint32_t a[4];
            ldmatrix_x4(a, smem_u32(sQ + (mb * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * LD + kk * 16 +
                                    (lane >> 4) * 8));
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                if (j < nt) {
                    uint32_t bb[2];
                    ldmatrix_x2(bb, smem_u32(sK + (j * 8 + (lane & 7)) * LD + kk * 16 + ((lane >> 3) & 1) * 8));
                    mma_bf16_16816(s[j], a, bb);
                }
            }
        }
        // Causal mask, softmax in fp32 (rows r0 and r1 of this thread).
        const int r0 = mb * 16 + gq, r1 = r0 + 8;
        float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            if (j < nt) {
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const int key = j * 8 + tig * 2 + (q & 1);
                    const int row = q < 2 ? r0 : r1;
                    if (key > row || key >= n) s[j][q] = -INFINITY;
                }
                m0 = fmaxf(m0, fmaxf(s[j][0], s[j][1]));
                m1 = fmaxf(m1, fmaxf(s[j][2], s[j][3]));
            }
        }
#pragma unroll
        for (int o = 1; o <= 2; o <<= 1) {
            m0 = fmaxf(m0, __shfl_xor_sync(0xffffffffu, m0, o));
            m1 = fmaxf(m1, __shfl_xor_sync(0xffffffffu, m1, o));
        }
        float l0 = 0.f, l1 = 0.f;
#pragma unroll
        for (int j = 0; j < 16; ++j) {
            if (j < nt) {
                s[j][0] = expf((s[j][0] - m0) * p.scale);
                s[j][1] = expf((s[j][1] - m0) * p.scale);
                s[j][2] = expf((s[j][2] - m1) * p.scale);
                s[j][3] = expf((s[j][3] - m1) * p.scale);
                l0 += s[j][0] + s[j][1];
                l1 += s[j][2] + s[j][3];
            }
        }
#pragma unroll
        for (int o = 1; o <= 2; o <<= 1) {
            l0 += __shfl_xor_sync(0xffffffffu, l0, o);
            l1 += __shfl_xor_sync(0xffffffffu, l1, o);
        }
        // O = P V over the key steps of 16 up to the block's last row.
        float acc[NTO][4];
#pragma unroll
        for (int j = 0; j < NTO; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
            if (kk <= mb) {
                uint32_t a[4];
                a[0] = pack_bf16x2(s[2 * kk][0], s[2 * kk][1]);
                a[1] = pack_bf16x2(s[2 * kk][2], s[2 * kk][3]);
                a[2] = pack_bf16x2(s[2 * kk + 1][0], s[2 * kk + 1][1]);
                a[3] = pack_bf16x2(s[2 * kk + 1][2], s[2 * kk + 1][3]);
#pragma unroll
                for (int jn = 0; jn < NTO; jn += 2) {
                    uint32_t bb[4];
                    ldmatrix_x4_trans(bb, smem_u32(sV + (kk * 16 + (lane & 7) + ((lane >> 3) & 1) * 8) * LD +
                                                   jn * 8 + (lane >> 4) * 8));
                    const uint32_t b0[2] = {bb[0], bb[1]}, b1[2] = {bb[2], bb[3]};
                    mma_bf16_16816(acc[jn], a, b0);
                    mma_bf16_16816(acc[jn + 1], a, b1);
                }
            }
        }
        // Normalise, stage the 16 rows in this warp's own Q rows, store 16-byte rows.
        const float i0 = 1.f / l0, i1 = 1.f / l1;
#pragma unroll
        for (int jn = 0; jn < NTO; ++jn) {
            const int col = jn * 8 + tig * 2;
            *reinterpret_cast<uint32_t*>(sQ + r0 * LD + col) = pack_bf16x2(acc[jn][0] * i0, acc[jn][1] * i0);
            *reinterpret_cast<uint32_t*>(sQ + r1 * LD + col) = pack_bf16x2(acc[jn][2] * i1, acc[jn][3] * i1);
        }
        __syncwarp();
        for (int i = lane; i < 16 * (DH / 8); i += 32) {
            const int rr = i / (DH / 8), c = (i - rr * (DH / 8)) * 8;
            const int row = mb * 16 + rr;
            if (row < n)
                *reinterpret_cast<uint4*>(p.out + (size_t)(t0 + row) * ostride + qoff + c) =
                    *reinterpret_cast<const uint4*>(sQ + row * LD + c);
        }
        __syncwarp();
    }
    pdl_trigger();   // the next kernel may be scheduled once every block got here or exited
}

template <int DH>
constexpr size_t attn_smem() {
    return (size_t)3 * kSeqMax * (DH + 8) * sizeof(__nv_bfloat16);
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

cudaError_t launch_attention(const AttnParams& p, int head_dim, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    if (p.S < 1 || p.S > kSeqMax || p.Hkv < 1 || p.Hq % p.Hkv) return cudaErrorInvalidValue;
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(attention_kernel<64>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)attn_smem<64>());
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(attention_kernel<128>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)attn_smem<128>());
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const dim3 grid(p.Hq, (p.T + p.S - 1) / p.S);
    cudaError_t e;
    if (head_dim == 64) e = launch_pdl(attention_kernel<64>, grid, dim3(128), attn_smem<64>(), st, p);
    else if (head_dim == 128) e = launch_pdl(attention_kernel<128>, grid, dim3(128), attn_smem<128>(), st, p);
    else return cudaErrorInvalidValue;
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
