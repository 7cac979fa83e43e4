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
            for (int j = 0; j < nj; ++j) {
                const float gj = p.topk_g[t * p.k + j];
                w[j] = p.renorm ? __fdiv_rn(gj, gs) : gj;
                pos[j] = p.pos_pair[t * p.k + j];
            }
        }
        const int psh = p.has_shared ? p.pos_sh[t] : -1;
        uint4* hrow = reinterpret_cast<uint4*>(p.h + (size_t)t * p.d);
        const uint4* brow = reinterpret_cast<const uint4*>(p.h_src + (size_t)t * p.d);
        for (int c = lane; c < nchunk; c += 32) {
            const uint4 hv = brow[c];
            float acc[8] = {bf16_lo(hv.x), bf16_hi(hv.x), bf16_lo(hv.y), bf16_hi(hv.y),
                            bf16_lo(hv.z), bf16_hi(hv.z), bf16_lo(hv.w), bf16_hi(hv.w)};
            for (int j = 0; j < nj; ++j) {
                const uint4 y = __ldg(reinterpret_cast<const uint4*>(p.Y + (size_t)pos[j] * p.d) + c);
                acc[0] = fmaf(w[j], bf16_lo(y.x), acc[0]);
                acc[1] = fmaf(w[j], bf16_hi(y.x), acc[1]);
                acc[2] = fmaf(w[j], bf16_lo(y.y), acc[2]);
                acc[3] = fmaf(w[j], bf16_hi(y.y), acc[3]);
                acc[4] = fmaf(w[j], bf16_lo(y.z), acc[4]);
                acc[5] = fmaf(w[j], bf16_hi(y.z), acc[5]);
                acc[6] = fmaf(w[j], bf16_lo(y.w), acc[6]);
                acc[7] = fmaf(w[j], bf16_hi(y.w), acc[7]);
            }
            if (psh >= 0) {
                const uint4 y = __ldg(reinterpret_cast<const uint4*>(p.Ysh + (size_t)psh * p.d) + c);
                acc[0] += bf16_lo(y.x);
                acc[1] += bf16_hi(y.x);
                acc[2] += bf16_lo(y.y);
                acc[3] += bf16_hi(y.y);
                acc[4] += bf16_lo(y.z);
                acc[5] += bf16_hi(y.z);
                acc[6] += bf16_lo(y.w);
                acc[7] += bf16_hi(y.w);
            }
            uint4 o;
            o.x = pack_bf16x2(acc[0], acc[1]);
            o.y = pack_bf16x2(acc[2], acc[3]);
            o.z = pack_bf16x2(acc[4], acc[5]);
            o.w = pack_bf16x2(acc[6], acc[7]);
            hrow[c] = o;
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
