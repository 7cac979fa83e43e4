// Kernel (b): compaction of the executed (token, slot) pairs by expert and of
// the tokens that run the shared expert, then a gather of their hidden rows.
//
// The order is a stable counting sort: pairs of expert e are laid out in
// increasing (t, j), experts in increasing e, and the shared-expert rows
// (tokens executed or skipped at this layer) follow in increasing t.  Alg. 2
// (Sec. V-E) removes exited tokens from the active set; only the survivors'
// pairs reach the expert FFN.
//
// Two passes over chunks of kChunk tokens: per-chunk bucket counts, then a
// scatter in which each chunk's block derives its base and the group offsets
// from all chunks' counts and each of its warps walks its 32 tokens in order,
// ranking equal buckets with __match_any_sync (one pass for a single chunk).
#include <mutex>
#include <string>

#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int kChunk = 256;

__global__ void __launch_bounds__(kChunk) count_kernel(const CompactParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    __shared__ int cnt[kMaxE + 1];
    const int nb = p.E + 1;
    for (int i = threadIdx.x; i < nb; i += blockDim.x) cnt[i] = 0;
    __syncthreads();
    const int t = blockIdx.x * kChunk + threadIdx.x;
    if (t < p.T) {
        const int a = p.action[t];
        if (a == 0)
            for (int j = 0; j < p.k; ++j) atomicAdd(&cnt[p.exp_sel[t * p.k + j]], 1);
        if (p.has_shared && (a == 0 || a == 1)) atomicAdd(&cnt[p.E], 1);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nb; i += blockDim.x) p.blk_counts[blockIdx.x * nb + i] = cnt[i];
}

// One block per chunk, one warp per 32 consecutive tokens of it.  The block
// first reads every chunk's counts: per bucket, the sum over the earlier chunks
// (this chunk's base) and over all chunks (the bucket total), and scans the
// totals into the group offsets (block 0 publishes them).  Each warp counts its
// pairs per bucket, the block turns the counts into per-warp starting
// positions (group offset + chunk base + the earlier warps' counts), and each
// warp then walks its pairs in (t, j) order, 32 at a time, ranking equal
// buckets with __match_any_sync.  Integer sums: the result does not depend on
// the order of the additions.  With a single chunk (T <= kChunk) the block
// counts its own pairs: no count kernel, and the bucket totals are the sums of
// the warps' counts.
constexpr int kScatWarps = kChunk / 32;

template <bool kSingle>
__global__ void __launch_bounds__(kChunk) scatter_kernel(const CompactParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    __shared__ int run[kScatWarps][kMaxE + 1];
    __shared__ int cbase[kMaxE + 1], total[kMaxE + 1], goff_s[kMaxE + 2];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nb = p.E + 1;
    for (int i = threadIdx.x; i < kScatWarps * nb; i += blockDim.x) run[i / nb][i % nb] = 0;
    // Chunk base and total per bucket: a warp per bucket, lanes over chunks.
    for (int e = warp; e < (kSingle ? 0 : nb); e += kScatWarps) {
        int pre = 0, all = 0;
        for (int b0 = 0; b0 < p.nblk; b0 += 32) {
            const int b = b0 + lane;
            const int c = b < p.nblk ? p.blk_counts[b * nb + e] : 0;
            all += c;
            pre += b < (int)blockIdx.x ? c : 0;
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            all += __shfl_xor_sync(0xffffffffu, all, o);
            pre += __shfl_xor_sync(0xffffffffu, pre, o);
        }
        if (lane == 0) {
            cbase[e] = pre;
            total[e] = all;
        }
    }
    __syncthreads();
    const int t0 = blockIdx.x * kChunk + warp * 32;
    const int tn = max(0, min(32, p.T - t0));
    const unsigned lt_mask = (1u << lane) - 1u;
    const int npairs = tn * p.k;
    // Pass 1: this warp's count per bucket.
    for (int q0 = 0; q0 < npairs; q0 += 32) {
        const int q = q0 + lane;
        int key = -1;
        if (q < npairs) {
            const int t = t0 + q / p.k;
            if (p.action[t] == 0) key = p.exp_sel[t * p.k + (q - (q / p.k) * p.k)];
        }
        const unsigned peers = __match_any_sync(0xffffffffu, key);
        if (key >= 0 && (peers & lt_mask) == 0) run[warp][key] += __popc(peers);
    }
    if (p.has_shared) {
        const bool take = lane < tn && (p.action[t0 + lane] == 0 || p.action[t0 + lane] == 1);
        const unsigned ball = __ballot_sync(0xffffffffu, take);
        if (lane == 0) run[warp][p.E] = __popc(ball);
    }
    __syncthreads();
    if (kSingle) {
        for (int e = threadIdx.x; e < nb; e += blockDim.x) {
            int all = 0;
            for (int w = 0; w < kScatWarps; ++w) all += run[w][e];
            cbase[e] = 0;
            total[e] = all;
        }
    }
    __syncthreads();
    if (warp == 0) {
        // Group offsets: exclusive prefix of the bucket totals.
        int base = 0;
        unsigned long long touched = 0;
        for (int e0 = 0; e0 < nb; e0 += 32) {
            const int e = e0 + lane;
            const int c = e < nb ? total[e] : 0;
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (e < nb) goff_s[e] = base + incl - c;
            touched += __popc(__ballot_sync(0xffffffffu, e < p.E && c > 0));
            base += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) goff_s[nb] = base;
        if (blockIdx.x == 0) {
            __syncwarp();
            for (int e = lane; e <= nb; e += 32) p.goff[e] = goff_s[e];
            if (lane == 0) {
                atomicAdd(&p.ctr->pairs_total, (unsigned long long)(base - total[p.E]));
                atomicAdd(&p.ctr->shared_rows, (unsigned long long)total[p.E]);
                atomicAdd(&p.ctr->experts_touched, touched);
                if (total[p.E] > 0) atomicAdd(&p.ctr->shared_touched, 1ull);
            }
        }
    }
    __syncthreads();
    // Per-warp starting positions: exclusive prefix over the warps, per bucket.
    for (int e = threadIdx.x; e < nb; e += blockDim.x) {
        int acc = goff_s[e] + cbase[e];
        for (int w = 0; w < kScatWarps; ++w) {
            const int c = run[w][e];
            run[w][e] = acc;
            acc += c;
        }
    }
    __syncthreads();
    // Pass 2: routed pairs.
    for (int q0 = 0; q0 < npairs; q0 += 32) {
        const int q = q0 + lane;
        int key = -1, code = -1;
        if (q < npairs) {
            const int t = t0 + q / p.k;
            const int j = q - (q / p.k) * p.k;
            code = t * p.k + j;
            if (p.action[t] == 0) key = p.exp_sel[code];
            else p.pos_pair[code] = -1;
        }
        const unsigned peers = __match_any_sync(0xffffffffu, key);
        if (key >= 0) {
            const int pos = run[warp][key] + __popc(peers & lt_mask);
            p.perm[pos] = code;
            p.pos_pair[code] = pos;
        }
        __syncwarp();
        if (key >= 0 && (peers & lt_mask) == 0) run[warp][key] += __popc(peers);
        __syncwarp();
    }
    // Shared-expert rows: executed or skipped tokens, by t.
    if (p.has_shared && tn > 0) {
        const int t = t0 + lane;
        bool take = false;
        if (lane < tn) {
            const int a = p.action[t];
            take = (a == 0 || a == 1);
            if (!take) p.pos_sh[t] = -1;
        }
        const unsigned ball = __ballot_sync(0xffffffffu, take);
        if (take) {
            const int pos = run[warp][p.E] + __popc(ball & lt_mask);
            p.perm[pos] = t;
            p.pos_sh[t] = pos - goff_s[p.E];
        }
    }
}

// Xp[row] = expert input of the row's token: bf16(h * r * gamma) with the
// pre-FFN RMSNorm, or h itself without it; one warp per row, gamma staged in
// shared memory once per block, kGU chunks of 16 bytes per lane in flight.
constexpr int kGU = 8;
constexpr int kMaxGatherD = 16384;   // gamma staged in shared memory (32 KB)

__global__ void __launch_bounds__(256) gather_kernel(const int32_t* __restrict__ perm,
                                                     const int32_t* __restrict__ goff, int E, int k,
                                                     int d, const __nv_bfloat16* __restrict__ h,
                                                     const float* __restrict__ rnorm,
                                                     const __nv_bfloat16* __restrict__ gamma,
                                                     __nv_bfloat16* __restrict__ Xp, int nseg) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    extern __shared__ uint4 sg[];      // gamma, d / 8 chunks
    const int nrows = goff[E + 1];
    const int routed = goff[E];
    const int lane = threadIdx.x & 31;
    const int nchunk = d >> 3;
    if (gamma) {
        const uint4* gv4 = reinterpret_cast<const uint4*>(gamma);
        for (int c = threadIdx.x; c < nchunk; c += blockDim.x) sg[c] = __ldg(gv4 + c);
        __syncthreads();
    }
    // A warp copies one of nseg segments of a row (nseg > 1 for decode-sized
    // batches, so that a row's loads are in flight together).
    const int seg_chunks = (nchunk + nseg - 1) / nseg;
    const long long nunits = (long long)nrows * nseg;
    for (long long unit = (blockIdx.x * blockDim.x + threadIdx.x) >> 5; unit < nunits;
         unit += (gridDim.x * blockDim.x) >> 5) {
        const int r = (int)(unit / nseg);
        const int cbeg = (int)(unit - (long long)r * nseg) * seg_chunks;
        const int cend = min(nchunk, cbeg + seg_chunks);
        const int code = perm[r];
        const int t = r < routed ? code / k : code;
        const uint4* __restrict__ src = reinterpret_cast<const uint4*>(h + (size_t)t * d);
        uint4* __restrict__ dst = reinterpret_cast<uint4*>(Xp + (size_t)r * d);
        const float rn = gamma ? rnorm[t] : 1.f;
        for (int c0 = cbeg + lane; c0 < cend; c0 += 32 * kGU) {
            uint4 hv[kGU];
#pragma unroll
            for (int u = 0; u < kGU; ++u)
                if (c0 + 32 * u < cend) hv[u] = src[c0 + 32 * u];
#pragma unroll
            for (int u = 0; u < kGU; ++u) {
                const int c = c0 + 32 * u;
                if (c >= cend) continue;
                if (!gamma) {
                    dst[c] = hv[u];
                    continue;
                }
                const uint4 gv = sg[c];
                uint4 o;
                o.x = pack_bf16x2(bf16_lo(hv[u].x) * rn * bf16_lo(gv.x), bf16_hi(hv[u].x) * rn * bf16_hi(gv.x));
                o.y = pack_bf16x2(bf16_lo(hv[u].y) * rn * bf16_lo(gv.y), bf16_hi(hv[u].y) * rn * bf16_hi(gv.y));
                o.z = pack_bf16x2(bf16_lo(hv[u].z) * rn * bf16_lo(gv.z), bf16_hi(hv[u].z) * rn * bf16_hi(gv.z));
                o.w = pack_bf16x2(bf16_lo(hv[u].w) * rn * bf16_lo(gv.w), bf16_hi(hv[u].w) * rn * bf16_hi(gv.w));
                dst[c] = o;
            }
        }
    }
}

}  // namespace

cudaError_t launch_compact(const CompactParams& p, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    cudaError_t e;
    if (p.nblk == 1) {
        e = launch_pdl(scatter_kernel<true>, dim3(1), dim3(kChunk), 0, st, p);
    } else {
        e = launch_pdl(count_kernel, dim3(p.nblk), dim3(kChunk), 0, st, p);
        if (e == cudaSuccess) e = launch_pdl(scatter_kernel<false>, dim3(p.nblk), dim3(kChunk), 0, st, p);
    }
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

cudaError_t launch_gather(const int32_t* perm, const int32_t* goff, int E, int k, int d,
                          const __nv_bfloat16* h, const float* rnorm, const __nv_bfloat16* gamma,
                          __nv_bfloat16* Xp, int max_rows, int num_sms, cudaStream_t st) {
    if (max_rows <= 0) return cudaSuccess;
    if (d > kMaxGatherD) return cudaErrorInvalidValue;
    const size_t smem = gamma ? (size_t)d * 2 : 0;
    static PerDevice occ;
    const int per_sm = occ.get([] {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, gather_kernel, 256, (size_t)kMaxGatherD * 2) !=
                cudaSuccess || n < 1)
            n = 1;
        return n;
    });
    // Decode-sized batches: one row segment (a step of kGU chunks per lane) per warp.
    const int steps = ((d >> 3) + 32 * kGU - 1) / (32 * kGU);
    const int nseg = max_rows <= 512 && steps > 1 ? steps : 1;
    long long want = ((long long)max_rows * nseg + 7) / 8;
    const int blocks = (int)(want < (long long)num_sms * per_sm ? want : (long long)num_sms * per_sm);
    const cudaError_t e = launch_pdl(gather_kernel, dim3(blocks), dim3(256), smem, st, perm, goff, E, k, d, h, rnorm,
                                     gamma, Xp, nseg);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe

// ---------------------------------------------------------------------------
// Compaction without any device allocation.
//
// Some callers cannot call cudaMalloc at all: code running inside an
// allocator's own callback, processes whose device memory is fully handed to
// another pool, or hosts that must not allocate during a captured or
// latency-critical section.  For them the per-chunk counts and bases of the
// compaction live in this file-scope device array instead of a handle's
// workspace.  Its size is fixed (about 132 KB); every GPU that loads the
// library holds it until the process exits.
namespace tmoe {
namespace {

constexpr int kNoAllocMaxT = 65536;
constexpr int kNoAllocMaxBlk = kNoAllocMaxT / kChunk;

struct NoAllocScratch {
    int32_t blk_counts[kNoAllocMaxBlk * (kMaxE + 1)];
    DevCounters ctr;
};

}  // namespace
}  // namespace tmoe

static __device__ __align__(256) unsigned char g_noalloc_scratch[sizeof(tmoe::NoAllocScratch)];

namespace {

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mu;
void* g_noalloc_ptr[kMaxDevices] = {nullptr};
unsigned long long g_noalloc_ctx[kMaxDevices] = {0};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Identity of the calling thread's current CUDA context (0 if the driver
// entry points are unavailable or no context is current).  A context made
// after cudaDeviceReset has a new identity, and the module holding the array
// is loaded again there, possibly at another address.
unsigned long long current_context_id(bool* available) {
    static CtxGetCurrentFn get_current = nullptr;
    static CtxGetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        void* q = nullptr;
        cudaDriverEntryPointQueryResult r1, r2;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &r1) == cudaSuccess &&
            r1 == cudaDriverEntryPointSuccess &&
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &q, 12000, cudaEnableDefault, &r2) == cudaSuccess &&
            r2 == cudaDriverEntryPointSuccess) {
            get_current = reinterpret_cast<CtxGetCurrentFn>(p);
            get_id = reinterpret_cast<CtxGetIdFn>(q);
        }
    });
    *available = get_current && get_id;
    if (!*available) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array on the current device.  The host-side
// symbol is only a stand-in, never a device address, so the address is looked
// up with cudaGetSymbolAddress at set-up: on the first call on each device,
// with that device current, and again only if the device's context has been
// replaced since (cudaDeviceReset), never on other calls.
trimmoe_status noalloc_scratch(tmoe::NoAllocScratch** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) {
        tmoe::set_global_error("compact_noalloc: no usable current CUDA device");
        return TRIMMOE_ERR_CUDA;
    }
    std::lock_guard<std::mutex> g(g_noalloc_mu);
    bool have_ids = false;
    const unsigned long long ctx = current_context_id(&have_ids);
    const bool stale = have_ids && (ctx == 0 || ctx != g_noalloc_ctx[dev]);
    if (!g_noalloc_ptr[dev] || stale) {
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess || !p) {
            tmoe::set_global_error(std::string("compact_noalloc: cudaGetSymbolAddress failed: ") +
                                   cudaGetErrorString(e));
            return TRIMMOE_ERR_CUDA;
        }
        g_noalloc_ptr[dev] = p;
        // The lookup makes the device's primary context current if none was.
        g_noalloc_ctx[dev] = have_ids ? current_context_id(&have_ids) : 0;
    }
    *out = static_cast<tmoe::NoAllocScratch*>(g_noalloc_ptr[dev]);
    return TRIMMOE_OK;
}

}  // namespace

extern "C" trimmoe_status trimmoe_compact_noalloc(const uint8_t* action, const uint8_t* exp_sel, int T,
                                                  int k, int E, int has_shared, int32_t* perm,
                                                  int32_t* group_off, int32_t* pos_pair, int32_t* pos_sh,
                                                  void* stream) {
    using namespace tmoe;
    if (T < 0 || T > kNoAllocMaxT) {
        set_global_error("compact_noalloc: T must be in [0, 65536] (size of the static scratch)");
        return TRIMMOE_ERR_ARG;
    }
    if (E < 1 || E > kMaxE || k < 1 || k > kMaxK || k > E) {
        set_global_error("compact_noalloc: need 1 <= E <= 128 and 1 <= k <= min(E, 8)");
        return TRIMMOE_ERR_ARG;
    }
    if (!action || !exp_sel || !perm || !group_off || !pos_pair || (has_shared && !pos_sh)) {
        set_global_error("compact_noalloc: NULL pointer");
        return TRIMMOE_ERR_ARG;
    }
    NoAllocScratch* s = nullptr;
    trimmoe_status rc = noalloc_scratch(&s);
    if (rc != TRIMMOE_OK) return rc;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    // Only the counters must start at zero; the counts are fully rewritten.
    if (cudaMemsetAsync(&s->ctr, 0, sizeof(DevCounters), st) != cudaSuccess) {
        set_global_error("compact_noalloc: cudaMemsetAsync failed");
        return TRIMMOE_ERR_CUDA;
    }
    if (T == 0) {
        if (cudaMemsetAsync(group_off, 0, (size_t)(E + 2) * sizeof(int32_t), st) != cudaSuccess) {
            set_global_error("compact_noalloc: cudaMemsetAsync failed");
            return TRIMMOE_ERR_CUDA;
        }
        return TRIMMOE_OK;
    }
    CompactParams cp;
    cp.T = T;
    cp.k = k;
    cp.E = E;
    cp.has_shared = has_shared ? 1 : 0;
    cp.nblk = (T + kChunk - 1) / kChunk;
    cp.action = action;
    cp.exp_sel = exp_sel;
    cp.blk_counts = s->blk_counts;
    cp.goff = group_off;
    cp.perm = perm;
    cp.pos_pair = pos_pair;
    cp.pos_sh = pos_sh;
    cp.ctr = &s->ctr;
    const cudaError_t e = launch_compact(cp, st);
    if (e != cudaSuccess) {
        set_global_error(std::string("compact_noalloc: ") + cudaGetErrorString(e));
        return TRIMMOE_ERR_CUDA;
    }
    return TRIMMOE_OK;
}
