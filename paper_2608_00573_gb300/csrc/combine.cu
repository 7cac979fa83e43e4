// Kernel (d): un-permute and gate-weighted combine with the residual path.
//
//   EXEC:  h[t] = bf16( b[t] + sum_j w_j * Y[pos(t, j)] (+ Ysh[t]) )
//   SKIP:  h[t] = bf16( b[t] + Ysh[t] )
//   EXIT / DEAD: untouched.
// The residual base b is h itself (the MoE step alone: then a skip without a
// shared expert is not touched either) or the post-attention state of the full
// block, which executed and skipped tokens carry on while an exiting token
// keeps the state that entered the layer.
// w_j are the router gates of the top-k slots, renormalised over the top-k
// when requested; a substitute expert takes its target's gate.  A skipped
// layer is the identity (residual) path of Sec. III-B; the shared expert is
// local and runs for every token that is still active (Sec. III-B).
// One warp per token, 16-byte loads and stores, fp32 accumulation in slot order.
#include "internal.cuh"

namespace tmoe {

namespace {

__global__ void __launch_bounds__(256) combine_kernel(const CombineParams p) {
    const int lane = threadIdx.x & 31;
    const int nchunk = p.d >> 3;
    for (int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; t < p.T;
         t += (gridDim.x * blockDim.x) >> 5) {
        const int a = p.action[t];
        if (a > 1 || (a == 1 && !p.has_shared && p.h_src == p.h)) continue;
        float w[kMaxK];
        int pos[kMaxK];
        int nj = 0;
        if (a == 0) {
            nj = p.k;
            float gs = 0.f;
            for (int j = 0; j < nj; ++j) gs = __fadd_rn(gs, p.topk_g[t * p.k + j]);
#pragma unroll
            for (int j = 0; j < kMaxK; ++j) {
                if (j < nj) {
                    const float gj = p.topk_g[t * p.k + j];
                    w[j] = p.renorm ? __fdiv_rn(gj, gs) : gj;
                    pos[j] = p.pos_pair[t * p.k + j];
                }
            }
        }
        const int psh = p.has_shared ? p.pos_sh[t] : -1;
        uint4* hrow = reinterpret_cast<uint4*>(p.h + (size_t)t * p.d);
        const uint4* brow = reinterpret_cast<const uint4*>(p.h_src + (size_t)t * p.d);
        // kU chunks of 16 bytes per lane at a time: every load of a step is in
        // flight before the first one is used.
        constexpr int kU = 4;
        for (int c0 = lane; c0 < nchunk; c0 += 32 * kU) {
            float acc[kU][8];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + 32 * u;
                const uint4 hv = c < nchunk ? brow[c] : make_uint4(0u, 0u, 0u, 0u);
                acc[u][0] = bf16_lo(hv.x); acc[u][1] = bf16_hi(hv.x);
                acc[u][2] = bf16_lo(hv.y); acc[u][3] = bf16_hi(hv.y);
                acc[u][4] = bf16_lo(hv.z); acc[u][5] = bf16_hi(hv.z);
                acc[u][6] = bf16_lo(hv.w); acc[u][7] = bf16_hi(hv.w);
            }
#pragma unroll
            for (int j = 0; j < kMaxK; ++j) {
                if (j >= nj) break;
                const uint4* yrow = reinterpret_cast<const uint4*>(p.Y + (size_t)pos[j] * p.d);
                uint4 y[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int c = c0 + 32 * u;
                    y[u] = c < nchunk ? __ldg(yrow + c) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    acc[u][0] = fmaf(w[j], bf16_lo(y[u].x), acc[u][0]);
                    acc[u][1] = fmaf(w[j], bf16_hi(y[u].x), acc[u][1]);
                    acc[u][2] = fmaf(w[j], bf16_lo(y[u].y), acc[u][2]);
                    acc[u][3] = fmaf(w[j], bf16_hi(y[u].y), acc[u][3]);
                    acc[u][4] = fmaf(w[j], bf16_lo(y[u].z), acc[u][4]);
                    acc[u][5] = fmaf(w[j], bf16_hi(y[u].z), acc[u][5]);
                    acc[u][6] = fmaf(w[j], bf16_lo(y[u].w), acc[u][6]);
                    acc[u][7] = fmaf(w[j], bf16_hi(y[u].w), acc[u][7]);
                }
            }
            if (psh >= 0) {
                const uint4* yrow = reinterpret_cast<const uint4*>(p.Ysh + (size_t)psh * p.d);
                uint4 y[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int c = c0 + 32 * u;
                    y[u] = c < nchunk ? __ldg(yrow + c) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    acc[u][0] += bf16_lo(y[u].x);
                    acc[u][1] += bf16_hi(y[u].x);
                    acc[u][2] += bf16_lo(y[u].y);
                    acc[u][3] += bf16_hi(y[u].y);
                    acc[u][4] += bf16_lo(y[u].z);
                    acc[u][5] += bf16_hi(y[u].z);
                    acc[u][6] += bf16_lo(y[u].w);
                    acc[u][7] += bf16_hi(y[u].w);
                }
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + 32 * u;
                if (c < nchunk) {
                    uint4 o;
                    o.x = pack_bf16x2(acc[u][0], acc[u][1]);
                    o.y = pack_bf16x2(acc[u][2], acc[u][3]);
                    o.z = pack_bf16x2(acc[u][4], acc[u][5]);
                    o.w = pack_bf16x2(acc[u][6], acc[u][7]);
                    hrow[c] = o;
                }
            }
        }
    }
}

}  // namespace

cudaError_t launch_combine(const CombineParams& p, int num_sms, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    int blocks = (p.T + 7) / 8;
    blocks = blocks < num_sms * 8 ? blocks : num_sms * 8;
    combine_kernel<<<blocks, 256, 0, st>>>(p);
    return cudaGetLastError();
}

}  // namespace tmoe
