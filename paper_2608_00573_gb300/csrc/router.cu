// Kernel (a0): router and exit-head dot products of a layer on the tensor cores.
//
//   z[t][e]     = r_t * sum_i h[t][i] * gamma_i * W_r[e][i] + b_r[e]     e < E   (Eq. 4 input)
//   z[t][E + c] = r_t * sum_i h[t][i] * W_x[c][i]            + b_x[c]     c < C   (Eq. 7 input)
// with r_t = 1/sqrt(mean_i h[t][i]^2 + eps) (1 without the pre-FFN RMSNorm).
// The columns i are split into ksplit ranges, one per blockIdx.y, so that the
// grid covers every SM several times even for small token counts; each block
// writes its partial sums (and partial sums of h^2), and the decision kernel
// adds the ranges in a fixed order before applying r and the bias.
//
// The router's gamma * W_r products are exact in fp32 and split exactly into
// two bf16 matrices (hi + lo), so two bf16 MMAs give the logits without
// rounding the normalised input.  Each 16-wide k step starts its MMA from zero
// and its partial is added to IEEE fp32 registers (__fadd_rn): the tensor
// core's own accumulation then only touches sums of 16-32 exact products, which
// keeps the logits at fp32 accuracy (the decisions compare them to 1e-5).
// mma.sync m16n8k16 (bf16 in, fp32 accumulate): the contraction is tiny (E + C
// outputs per token) and the kernel is bound by streaming h from HBM, so the
// tensor cores only remove the per-element unpack/FMA instruction cost.
// One block = 64 tokens (4 warps x 16), d streamed in 64-column slabs through
// a 4-stage cp.async ring in padded shared memory, ldmatrix fragments; up to
// 128 output rows per pass over h.
// Dead tokens are zero-filled without reading HBM.
#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int kTok = 64;
constexpr int kKS = 64;
constexpr int kPad = 72;          // padded smem row (bf16): conflict-free ldmatrix
constexpr int kStages = 4;
constexpr int kNG = 128;          // largest number of outputs per pass (16 n-tiles of 8)

// NT: n-tiles of 8 outputs held in registers per pass (8 or 16).
template <int NT>
__global__ void __launch_bounds__(128) router_kernel(const RouterParams p) {
    extern __shared__ __align__(16) uint8_t sm[];
    const int NG = p.ng;                       // padded rows per pass (<= kNG, multiple of 8)
    const int NL = p.nl;                       // padded rows with a lo part (<= NG)
    __nv_bfloat16* sA = reinterpret_cast<__nv_bfloat16*>(sm);
    __nv_bfloat16* sBh = sA + kStages * kTok * kPad;
    __nv_bfloat16* sBl = sBh + kStages * NG * kPad;
    __shared__ float ssq[kTok];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int t0 = blockIdx.x * kTok;
    const int nslab_all = p.d / kKS;
    const int nslab = nslab_all / p.ksplit;
    const int slab0 = blockIdx.y * nslab;
    float* zpart = p.zpart + (size_t)blockIdx.y * p.T * p.zs;
    float* sqpart = p.sqpart + (size_t)blockIdx.y * p.T;
    const int g = lane >> 2, tig = lane & 3;

    for (int ng0 = 0; ng0 < p.n_out; ng0 += NG) {
        const int nrows = min(NG, p.n_out - ng0);
        const int ntile = (nrows + 7) >> 3;
        const bool any_lo = ng0 < p.n_lo;
        float sq = 0.f;
        float acc[NT][4];
#pragma unroll
        for (int j = 0; j < NT; ++j) acc[j][0] = acc[j][1] = acc[j][2] = acc[j][3] = 0.f;

        auto load_slab = [&](int s) {
            const int buf = s % kStages;
            const int sg = slab0 + s;                 // global slab index
            for (int i = tid; i < kTok * (kKS / 8); i += 128) {
                const int r = i >> 3, c = i & 7;
                const int t = t0 + r;
                const bool ok = t < p.T && p.alive[t];
                const __nv_bfloat16* src = p.h + (size_t)(ok ? t : 0) * p.d + sg * kKS + c * 8;
                cp_async16(smem_u32(sA + (buf * kTok + r) * kPad + c * 8), src, ok ? 16 : 0);
            }
            for (int i = tid; i < NG * (kKS / 8); i += 128) {
                const int r = i >> 3, c = i & 7;
                const bool ok = r < nrows;
                const size_t off = (size_t)(ng0 + (ok ? r : 0)) * p.d + sg * kKS + c * 8;
                cp_async16(smem_u32(sBh + (buf * NG + r) * kPad + c * 8), p.Bhi + off, ok ? 16 : 0);
                if (any_lo && r < NL) {
                    const bool okl = ok && (ng0 + r) < p.n_lo;
                    cp_async16(smem_u32(sBl + (buf * NL + r) * kPad + c * 8), p.Blo + off, okl ? 16 : 0);
                }
            }
        };

        for (int s = 0; s < kStages - 1; ++s) {
            if (s < nslab) load_slab(s);
            cp_async_commit();
        }
        for (int s = 0; s < nslab; ++s) {
            cp_async_wait<kStages - 2>();
            __syncthreads();
            if (s + kStages - 1 < nslab) load_slab(s + kStages - 1);
            cp_async_commit();
            const int buf = s % kStages;
            const __nv_bfloat16* A = sA + buf * kTok * kPad;
            if (ng0 == 0) {                     // sum of squares for the RMS factor
                const __nv_bfloat16* row = A + (tid >> 1) * kPad + (tid & 1) * 32;
#pragma unroll
                for (int q = 0; q < 32; q += 8) {
                    const uint4 v = *reinterpret_cast<const uint4*>(row + q);
                    const float f[8] = {bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y),
                                        bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w)};
#pragma unroll
                    for (int u = 0; u < 8; ++u) sq = fmaf(f[u], f[u], sq);
                }
            }
#pragma unroll
            for (int kk = 0; kk < kKS / 16; ++kk) {
                uint32_t a[4];
                const int ar = warp * 16 + (lane & 7) + ((lane >> 3) & 1) * 8;
                const int ac = kk * 16 + (lane >> 4) * 8;
                ldmatrix_x4(a, smem_u32(A + ar * kPad + ac));
                const int br = (lane & 7);
                const int bc = kk * 16 + ((lane >> 3) & 1) * 8;
#pragma unroll
                for (int j = 0; j < NT; ++j) {
                    if (j < ntile) {
                        uint32_t b[2];
                        float part[4] = {0.f, 0.f, 0.f, 0.f};
                        ldmatrix_x2(b, smem_u32(sBh + (buf * NG + j * 8 + br) * kPad + bc));
                        mma_bf16_16816(part, a, b);
                        if (ng0 + j * 8 < p.n_lo) {
                            ldmatrix_x2(b, smem_u32(sBl + (buf * NL + j * 8 + br) * kPad + bc));
                            mma_bf16_16816(part, a, b);
                        }
#pragma unroll
                        for (int q = 0; q < 4; ++q) acc[j][q] = __fadd_rn(acc[j][q], part[q]);
                    }
                }
            }
        }
        cp_async_wait<0>();
        if (ng0 == 0) {
            sq += __shfl_xor_sync(0xffffffffu, sq, 1);
            if ((tid & 1) == 0) ssq[tid >> 1] = sq;
        }
        __syncthreads();
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int r = warp * 16 + g + half * 8;
            const int t = t0 + r;
            if (t >= p.T || !p.alive[t]) continue;
            if (ng0 == 0 && tig == 0) sqpart[t] = ssq[r];
            float* zrow = zpart + (size_t)t * p.zs;
#pragma unroll
            for (int j = 0; j < NT; ++j) {
                if (j < ntile) {
#pragma unroll
                    for (int q = 0; q < 2; ++q) {
                        const int col = ng0 + j * 8 + tig * 2 + q;
                        if (col < p.n_out) zrow[col] = acc[j][half * 2 + q];
                    }
                }
            }
        }
        __syncthreads();
    }
}

}  // namespace

size_t router_smem_bytes(int ng, int nl) {
    return (size_t)kStages * (kTok + ng + nl) * kPad * sizeof(__nv_bfloat16);
}

int router_lo_rows(int n_lo, int ng) {
    const int r = ((n_lo + 7) / 8) * 8;
    return r < ng ? r : ng;
}

// Column ranges per launch: a power of two dividing d/64, chosen so that the
// grid has at least about four blocks per SM.
int router_ksplit(int T, int d, int num_sms) {
    const int nslab = d / kKS;
    const int tiles = (T + kTok - 1) / kTok;
    int ks = 1;
    while (ks < nslab && (long long)tiles * ks < 4ll * num_sms && nslab % (ks * 2) == 0) ks *= 2;
    return ks;
}

int router_pass_rows(int n_out) {
    const int r = ((n_out + 7) / 8) * 8;
    return r < kNG ? r : kNG;
}

cudaError_t launch_router(const RouterParams& p, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    if (p.d % kKS || p.ksplit < 1 || (p.d / kKS) % p.ksplit) return cudaErrorInvalidValue;
    const size_t smem = router_smem_bytes(p.ng, p.nl);
    static bool attr_set = false;
    if (!attr_set) {
        cudaError_t e = cudaFuncSetAttribute(router_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)router_smem_bytes(kNG, kNG));
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(router_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                     (int)router_smem_bytes(kNG, kNG));
        if (e != cudaSuccess) return e;
        attr_set = true;
    }
    const dim3 grid((p.T + kTok - 1) / kTok, p.ksplit);
    if (p.ng <= 64) router_kernel<8><<<grid, 128, smem, st>>>(p);
    else router_kernel<16><<<grid, 128, smem, st>>>(p);
    return cudaGetLastError();
}

}  // namespace tmoe
