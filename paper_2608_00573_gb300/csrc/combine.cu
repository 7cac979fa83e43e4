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
// One warp per token, 16-byte loads and stores, fp32 accumulation in slot order
// (residual base, then w_j * Y_j for j ascending, then the shared row).
#include "internal.cuh"

namespace tmoe {

namespace {

// KT: slots held in registers (k <= KT).  All loads of one step (the residual
// base, every slot's Y row and the shared expert's row, kU chunks of 16 bytes
// per lane each) are issued before the first one is used.  A warp takes one
// segment of nseg of a token's row: the whole row (nseg = 1) for large
// batches, one step of it per warp for decode-sized ones, so that the row's
// loads are in flight at once rather than one step after another.
template <int KT>
__global__ void __launch_bounds__(256) combine_kernel(const CombineParams p, int nseg) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    constexpr int kU = KT <= 2 ? 4 : 2;
    const int lane = threadIdx.x & 31;
    const int nchunk = p.d >> 3;
    const int seg_chunks = (nchunk + nseg - 1) / nseg;
    const long long nunits = (long long)p.T * nseg;
    for (long long unit = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; unit < nunits;
         unit += (gridDim.x * blockDim.x) >> 5) {
        const int t = (int)(unit / nseg);
        const int cbeg = (int)(unit - (long long)t * nseg) * seg_chunks;
        const int cend = min(nchunk, cbeg + seg_chunks);
        const int a = p.action[t];
        if (a > 1 || (a == 1 && !p.has_shared && p.h_src == p.h)) continue;
        float w[KT];
        const uint4* yrow[KT];
        const int nj = a == 0 ? p.k : 0;
        if (a == 0) {
            float gs = 0.f;
            for (int j = 0; j < nj; ++j) gs = __fadd_rn(gs, p.topk_g[t * p.k + j]);
#pragma unroll
            for (int j = 0; j < KT; ++j) {
                if (j < nj) {
                    const float gj = p.topk_g[t * p.k + j];
                    w[j] = p.renorm ? __fdiv_rn(gj, gs) : gj;
                    yrow[j] = reinterpret_cast<const uint4*>(p.Y + (size_t)p.pos_pair[t * p.k + j] * p.d);
                }
            }
        }
        const int psh = p.has_shared ? p.pos_sh[t] : -1;
        const uint4* srow = reinterpret_cast<const uint4*>(p.Ysh + (size_t)(psh >= 0 ? psh : 0) * p.d);
        uint4* hrow = reinterpret_cast<uint4*>(p.h + (size_t)t * p.d);
        const uint4* brow = reinterpret_cast<const uint4*>(p.h_src + (size_t)t * p.d);
        for (int c0 = cbeg + lane; c0 < cend; c0 += 32 * kU) {
            uint4 hv[kU], yv[KT][kU], sv[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + 32 * u;
                hv[u] = c < cend ? brow[c] : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int j = 0; j < KT; ++j)
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int c = c0 + 32 * u;
                    yv[j][u] = (j < nj && c < cend) ? __ldg(yrow[j] + c) : make_uint4(0u, 0u, 0u, 0u);
                }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + 32 * u;
                sv[u] = (psh >= 0 && c < cend) ? __ldg(srow + c) : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const int c = c0 + 32 * u;
                if (c >= cend) continue;
                const uint32_t hw[4] = {hv[u].x, hv[u].y, hv[u].z, hv[u].w};
                uint32_t ow[4];
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    float lo = bf16_lo(hw[q]), hi = bf16_hi(hw[q]);
#pragma unroll
                    for (int j = 0; j < KT; ++j) {
                        if (j < nj) {
                            const uint32_t yw = q == 0 ? yv[j][u].x : q == 1 ? yv[j][u].y : q == 2 ? yv[j][u].z : yv[j][u].w;
                            lo = fmaf(w[j], bf16_lo(yw), lo);
                            hi = fmaf(w[j], bf16_hi(yw), hi);
                        }
                    }
                    if (psh >= 0) {
                        const uint32_t sw = q == 0 ? sv[u].x : q == 1 ? sv[u].y : q == 2 ? sv[u].z : sv[u].w;
                        lo += bf16_lo(sw);
                        hi += bf16_hi(sw);
                    }
                    ow[q] = pack_bf16x2(lo, hi);
                }
                hrow[c] = make_uint4(ow[0], ow[1], ow[2], ow[3]);
            }
        }
    }
}

// Row segments per token: one per warp step of kU chunks for decode-sized
// batches (at most 256 tokens), the whole row otherwise.
int combine_segments(int T, int d, int kU) {
    if (T > 256) return 1;
    const int steps = ((d >> 3) + 32 * kU - 1) / (32 * kU);
    return steps > 1 ? steps : 1;
}

template <int KT>
int combine_grid(int T, int num_sms) {
    static PerDevice occ;
    const int per_sm = occ.get([] {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, combine_kernel<KT>, 256, 0) != cudaSuccess || n < 1)
            n = 1;
        return n;
    });
    const int want = (T + 7) / 8;
    const int cap = num_sms * per_sm;
    return want < cap ? want : cap;
}

}  // namespace

cudaError_t launch_combine(const CombineParams& p, int num_sms, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    cudaError_t e;
    const int kU = p.k <= 2 ? 4 : 2;                  // combine_kernel's chunks per lane and step
    const int nseg = combine_segments(p.T, p.d, kU);
    const int units = p.T * nseg;
    if (p.k <= 1)
        e = launch_pdl(combine_kernel<1>, dim3(combine_grid<1>(units, num_sms)), dim3(256), 0, st, p, nseg);
    else if (p.k <= 2)
        e = launch_pdl(combine_kernel<2>, dim3(combine_grid<2>(units, num_sms)), dim3(256), 0, st, p, nseg);
    else if (p.k <= 4)
        e = launch_pdl(combine_kernel<4>, dim3(combine_grid<4>(units, num_sms)), dim3(256), 0, st, p, nseg);
    else
        e = launch_pdl(combine_kernel<kMaxK>, dim3(combine_grid<kMaxK>(units, num_sms)), dim3(256), 0, st, p, nseg);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
