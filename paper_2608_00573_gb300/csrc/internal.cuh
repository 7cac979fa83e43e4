// Internal declarations of the sm_103a TrimMoE library: the handle, kernel
// parameter blocks, launchers and the inline-PTX helpers (mbarrier, TMA,
// tcgen05) the kernels share.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>
#include <string>
#include <utility>

#include "../../include/trimmoe.h"

namespace tmoe {

constexpr int kMaxE = 128;
constexpr int kMaxK = 8;
constexpr int kMaxM = 16;
constexpr int kMaxH = 6;
constexpr int kMaxC = 256;
constexpr int kMaxCand = 64;        // (1 + n_sub) * M with n_sub <= 3, M <= 16
constexpr int kMaxME = 1024;        // look-ahead table entries per token
constexpr size_t kMaxIntervals = 4096;            // shared look-ahead tables per depth and layer
constexpr size_t kMaxTabFloats = (size_t)16 << 20; // 64 MB of shared look-ahead tables
constexpr size_t kMaxAllTabFloats = (size_t)64 << 20; // every layer's tables at once: up to 256 MB
constexpr int kGateUp = 128;        // W13 gate/up row interleave

// Device error codes (first one wins); the public TRIMMOE_DEVERR_* values.
enum : int { ERR_NONE = TRIMMOE_DEVERR_NONE, ERR_TIMEOUT_PRODUCER = TRIMMOE_DEVERR_GEMM_PRODUCER,
             ERR_TIMEOUT_MMA = TRIMMOE_DEVERR_GEMM_MMA, ERR_TIMEOUT_EPI = TRIMMOE_DEVERR_GEMM_EPILOGUE,
             ERR_TIMEOUT_ROUTER = TRIMMOE_DEVERR_ROUTER, ERR_TIMEOUT_ATTN = TRIMMOE_DEVERR_ATTENTION,
             ERR_TIMEOUT_SELFTEST = TRIMMOE_DEVERR_SELFTEST };

// Device-side counters (trimmoe_stats_t is assembled from these).  The handle
// keeps kCtrCopies copies, each on its own cache lines; a block of the
// decision kernel adds to copy blockIdx.x % kCtrCopies so that the atomics of
// different blocks do not queue on one line, and the host sums the copies.
constexpr int kCtrCopies = 32;
struct __align__(256) DevCounters {
    unsigned long long layer_tokens, exec_tokens, skipped, exited;
    unsigned long long pairs_local_exact, pairs_local_sub, pairs_remote_exact, pairs_remote_sub;
    unsigned long long shared_rows, remote_hops, pairs_total;
    unsigned long long experts_touched, shared_touched;   // (layer, expert) groups with work
    unsigned long long lookahead_shared;                  // decisions that read a shared look-ahead table
    double delay_ms;
    unsigned int max_budget_ratio_bits;   // non-negative float bits, atomicMax-able
};
static_assert(sizeof(DevCounters) == 256, "counter copies on separate cache lines");

// Per-layer decision tables on the device (built at create).
struct DevTables {
    const uint8_t* cand_m;   // flat candidate lists, all layers: server of candidate
    const uint8_t* cand_k;   // expert of candidate
    const float* cand_Q;     // substitution loss Q_l(r, k) (Eq. 3)
    const int* cand_off;     // [N][E+1] start of target r's list in the flat arrays
    const float* ctab;       // [N][M][M] omega_T * (d(m -> m') / d_ref) (Eq. 30-31)
    int max_layer_cand;      // largest number of candidates of one layer
    const float* trans;      // [M][M]
    const float* comp;       // [N][M]
    const float* P;          // [N-1][E][E]
    const float* theta;      // [N]
    const float* lambda;     // [N]
    const float* eps;        // [N]
};

// Router and exit-head partial logits of one layer (kernel a0), split over d:
// unit (tile, y) covers tokens [128 tile, 128 tile + 128) and columns
// [y*d/ksplit, (y+1)*d/ksplit); the hidden rows come through a tensor map
// passed beside these parameters.
struct RouterParams {
    int T, d;
    int n_out;                  // E + C logits per token
    int n_lo;                   // leading rows with a lo part (E)
    int ng;                     // rows per pass (multiple of 8, <= 128)
    int nl;                     // rows of the lo part staged per pass (multiple of 8, <= ng)
    int zs;                     // row stride of zpart
    int ksplit;                 // number of column ranges
    const __nv_bfloat16* h;
    const uint8_t* alive;
    const __nv_bfloat16* Bhi;   // [n_out][d] hi(gamma * W_r) then W_x of the previous layer
    const __nv_bfloat16* Blo;   // [E][d] lo(gamma * W_r)
    float* zpart;               // [T][ksplit][zs] partial dot products
    float* sqpart;              // [T][ksplit] partial sums of h^2
    int* err;                   // device error word (bounded waits)
};

struct DecideParams {
    int layer, T, N, d, E, k, C, M, H;
    float omega_T, omega_D, d_ref;
    const float* zpart;         // [T][ksplit][zs] partial router then exit-head dot products
    const float* sqpart;        // [T][ksplit] partial sums of h^2
    const float* sqpart_x;      // [T][ksplit] partial sums of the exit head's input^2 (NULL: sqpart)
    const float* bias;          // [E + C] router then exit-head biases of this layer
    int zs, ksplit;
    int use_norm;
    float norm_eps;
    float* rnorm;               // [T] RMS factor r (written when use_norm)
    int has_head;               // exit head of the previous layer available (layer > 0)
    int n_cent;                 // K_c centroids (Eq. 36), 0 = no exit prediction
    const float* cnorm;         // [K_c] centroid norms of this layer
    const int16_t* lhat_tab;    // [K_c] rounded average exit layer of each centroid
    int16_t* lhat_out;          // [T] predicted exit layer (may be NULL)
    // Shared look-ahead tables of the layer (Dbar = Dbar[0]): one per interval
    // between consecutive thresholds thr[0..n_thr) of the window and per depth
    // dmin..top_full, laid out [depth - dmin][interval][M*E].
    const float* phi_tabs;      // NULL: every token computes its own table
    const float* dbar_shared;
    const float* thr;           // sorted distinct Q and eps of layers l+1 .. l+top_full
    int n_thr;
    int dmin;
    float* phi_tabs_out;        // written by the shared-table kernel
    float* dbar_shared_out;
    // Per-token look-ahead scratch in global memory (one slot per resident
    // token group), used when the layer has shared tables (most tokens then
    // read a table and the scratch is rarely touched); NULL: in shared memory.
    float* la_scratch;
    // Offline-stage calibration counts (Algorithm 1), accumulated when calib != 0.
    int calib;
    int16_t* prev_target;       // [T] slot-0 target at the previous layer, -1 none
    unsigned long long* c_trans;   // [N-1][E][E]
    unsigned long long* c_alive;   // [N]
    unsigned long long* c_resid;   // [N][M]
    unsigned long long* c_act;     // [N][E]
    unsigned long long* c_above;   // [N][E]
    uint8_t* s;
    float* Dhat;
    const float* Dbar;
    const float* pJ;
    uint8_t* alive;
    uint8_t* last_exec;
    float* xi_last;
    int16_t* exit_layer;
    int32_t* topk_idx;
    float* topk_g;
    float* I_out;
    float* xi_out;
    uint8_t* action;
    uint8_t* exp_sel;
    uint8_t* srv_sel;
    DevTables tab;
    DevCounters* ctr;
};

struct CompactParams {
    int T, k, E, has_shared, nblk;
    const uint8_t* action;
    const uint8_t* exp_sel;
    int32_t* blk_counts;   // [nblk][E+1]
    int32_t* goff;         // [E+2]
    int32_t* perm;         // [T*k + T]
    int32_t* pos_pair;     // [T*k]
    int32_t* pos_sh;       // [T]
    DevCounters* ctr;
};

struct GemmLaunch {
    const CUtensorMap* tmA;
    const CUtensorMap* tmB;
    // Non-null: run the CTA-pair kernel, B loaded in 128-row boxes through this
    // map (launches whose groups are large; requires ksplit <= 1).
    const CUtensorMap* tmB_pair;
    // Non-zero (with tmB_pair): run the transposed pair kernel instead, the
    // weights on the M side of the MMA and the group's tokens on the N side
    // (STORE or RELU epilogues; ksplit <= 1).
    int transposed;
    const int* goff;
    int first_group, ngroups, a_rebase, out_rebase;
    int K, n_tiles_n, b_rows_per_group, epi_mode;
    __nv_bfloat16* out;
    int ldo;
    int* err;
    const __nv_bfloat16* res;   // EPI_RESID: residual rows (same row index as out)
    int ldr;
    const float2* rope;         // EPI_ROPE: (cos, sin) [rope_S][rope_dh/2]
    int rope_S, rope_dh, n_rot; // sequence length, head dim, leading columns that rotate
    // EPI_ROPE: the columns past n_rot (the value heads, vt_rows of them) are
    // stored transposed per sequence instead: vt[(seq * vt_rows + col - n_rot)
    // * kVtSlots + pos] for the token at position pos of sequence seq.
    __nv_bfloat16* vt;
    int vt_rows;
    // Split over K (ksplit > 1): each (tile, range) writes its fp32 partial
    // sums to partial[ks][row][col] (ldp columns, pstride floats per range) and
    // splitk_finish adds the ranges in order and applies the epilogue.
    int ksplit;
    float* partial;
    int ldp;
    size_t pstride;
    // Transposed pair kernel: launch-wide tile counter, zero when the launch
    // starts (each launch of a forward has its own, zeroed at the forward's
    // start).  Null: a static tile order.
    int* sched;
};

enum : int { EPI_STORE = 0, EPI_SWIGLU = 1, EPI_RELU = 2, EPI_RESID = 3, EPI_ROPE = 4 };

// Key slots per sequence in the transposed value buffer (the longest sequence).
constexpr int kVtSlots = 128;

// Parameters of the rotary (q/k/v projection) epilogue, see GemmLaunch.
struct RopeEpi {
    const float2* cs;
    int S, dh, n_rot;
    __nv_bfloat16* vt;
    int vt_rows;
};

// Attention sublayer of the full block (kernels e).
struct AttnParams {
    int T, d, S, Hq, Hkv, nqkv;
    float norm_eps, scale;
    const __nv_bfloat16* h;       // [T][d] state entering the layer
    const __nv_bfloat16* gamma;   // [d] RMSNorm weights of the sublayer
    __nv_bfloat16* a;             // [T][d] normalised input of the q/k/v projection
    int* goff;                    // [2] {0, T}: the projections' single GEMM group
    const __nv_bfloat16* qkv;     // [T][nqkv] query heads, key heads (rotated), value heads
    __nv_bfloat16* out;           // [T][Hq*Dh] attention output
    int* err;                     // device error word (bounded waits)
};

struct CombineParams {
    int T, d, k, renorm, has_shared;
    __nv_bfloat16* h;              // output rows (executed and skipped tokens)
    const __nv_bfloat16* h_src;    // residual base: h itself, or the post-attention state
    const uint8_t* action;
    const float* topk_g;
    const int32_t* pos_pair;
    const int32_t* pos_sh;
    const __nv_bfloat16* Y;
    const __nv_bfloat16* Ysh;
};

struct FeedbackParams {
    int T, N, user_size, users;
    float eta, p_min;
    float* pJ;
    const uint8_t* alive;
    const int16_t* exit_layer;
    const float* xi_last;
    const float* Dhat;
    const float* Dbar;
    double* util;       // [users]
    int* updated;       // [users]
    double* result;     // [2]: mean utilisation, users updated
};

// Launchers (one translation unit each).
// Tensor maps (64-column boxes, 128-byte swizzle): tmA the hidden rows [T][d]
// in 128-row boxes, tmBhi / tmBlo the pass's weight rows in ng / nl-row boxes.
cudaError_t launch_router(const CUtensorMap* tmA, const CUtensorMap* tmBhi, const CUtensorMap* tmBlo,
                          const RouterParams& p, int num_sms, cudaStream_t st);
int router_lo_rows(int n_lo, int ng);
int router_pass_rows(int n_out);
int router_ksplit(int T, int d, int n_out, int num_sms);
cudaError_t launch_decide(const DecideParams& p, int num_sms, cudaStream_t st);
size_t decide_smem_bytes(int E, int C, int M, int max_layer_cand);
size_t decide_la_scratch_floats(int E, int M, int max_layer_cand, int num_sms);
cudaError_t launch_lookahead_shared(const DecideParams& p, int n_depth, cudaStream_t st);
// Placement of one layer's shared look-ahead tables when every layer's tables
// are computed in one launch: thresholds p.thr[thr_off .. thr_off + n_thr),
// n_depth depths, tables from p.phi_tabs_out + tab_off.
struct LaLayer {
    int thr_off, n_thr, n_depth, tab_off;
};
cudaError_t launch_lookahead_all(const DecideParams& p, const LaLayer* layers, int n_layers, int max_thr,
                                 int max_depth, cudaStream_t st);
cudaError_t launch_compact(const CompactParams& p, cudaStream_t st);
cudaError_t launch_gather(const int32_t* perm, const int32_t* goff, int E, int k, int d,
                          const __nv_bfloat16* h, const float* rnorm, const __nv_bfloat16* gamma,
                          __nv_bfloat16* Xp, int max_rows, int num_sms, cudaStream_t st);
cudaError_t launch_grouped_gemm(const GemmLaunch& g, int num_sms, cudaStream_t st);
cudaError_t launch_splitk_finish(const GemmLaunch& g, int num_sms, cudaStream_t st);
int grouped_gemm_ksplit(int est_tiles, int nkb, int num_sms);
int grouped_gemm_pair_clusters(int num_sms);
size_t grouped_gemm_smem_bytes();
cudaError_t launch_combine(const CombineParams& p, int num_sms, cudaStream_t st);
cudaError_t launch_attn_norm(const AttnParams& p, int num_sms, cudaStream_t st);
// tm_qkv: the q/k/v rows [T][nqkv] in 128-row x 64-column boxes, 128-byte swizzle.
cudaError_t launch_attention(const AttnParams& p, const CUtensorMap* tm_qkv, const CUtensorMap* tm_vt, int head_dim,
                             int num_sms, cudaStream_t st);
cudaError_t launch_feedback(const FeedbackParams& p, cudaStream_t st);
cudaError_t launch_watchdog_selftest(int* err, uint64_t limit_ns, cudaStream_t st);

// Programmatic dependent launch.  The library's kernels are launched with
// programmatic stream serialisation: a kernel may be scheduled while the
// preceding grid in its stream is still finishing, runs its independent
// prologue, then waits (pdl_wait) for that grid to complete and its memory to be
// visible before touching anything written upstream.  Single-wave and
// persistent kernels let the next grid be scheduled right after their wait
// (pdl_trigger), multi-wave kernels only when each block is done, so that
// waiting blocks never take the room of their later waves.  After a launch
// without the attribute pdl_wait returns at once.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);
}

// Launch set-up kept per device: function attributes (dynamic shared memory
// limits) belong to a device's context and occupancy figures are per device,
// so one process-wide flag would skip the set-up on a second device.  get()
// runs f once for the current device under a lock and caches its result; with
// only_zero the result is cached only when it is 0 (cudaSuccess), so a failed
// set-up is tried again on the next call.
class PerDevice {
  public:
    static constexpr int kMaxDevices = 64;
    template <class F>
    int get(F&& f, bool only_zero = false) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return f();
        if (done_[dev].load(std::memory_order_acquire)) return val_[dev];
        std::lock_guard<std::mutex> g(mu_);
        if (done_[dev].load(std::memory_order_relaxed)) return val_[dev];
        const int v = f();
        if (!only_zero || v == 0) {
            val_[dev] = v;
            done_[dev].store(true, std::memory_order_release);
        }
        return v;
    }

  private:
    std::mutex mu_;
    std::atomic<bool> done_[kMaxDevices] = {};
    int val_[kMaxDevices] = {};
};

// Error text for calls made without a handle (read by trimmoe_last_error(NULL)).
void set_global_error(const std::string& msg);

// ------------------------------------------------------------------ PTX

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ uint64_t globaltimer_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

// Bounded wait: gives up after limit_ns (kTimeoutNs by default), raising the
// CTA abort flag and the device error word; also returns early once another
// role has aborted.
constexpr uint64_t kTimeoutNs = 2000000000ull;

__device__ __forceinline__ bool mbar_wait_bounded(uint32_t bar, uint32_t parity, volatile int* abort_flag,
                                                  int* err, int code, uint64_t limit_ns = kTimeoutNs) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = globaltimer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (globaltimer_ns() - t0 > limit_ns) {
            *abort_flag = 1;
            atomicCAS(err, 0, code);
            return false;
        }
    }
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap* tm, int x, int y,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void prefetch_tmap(const CUtensorMap* tm) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(tm)) : "memory");
}

__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

// D[tmem] (+)= A[smem] * B[smem]^T, kind::f16 (bf16 in, fp32 accumulate).
__device__ __forceinline__ void tc_mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                            uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive (once) on an mbarrier when all previously issued MMAs have completed.
__device__ __forceinline__ void tc_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// ---- CTA pairs (cluster of two, tcgen05 cta_group::2) -----------------------
__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Arrive on an mbarrier of another CTA of the cluster (cluster address from mapa).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t bar_cluster) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}

__device__ __forceinline__ void st_shared_cluster_u32(uint32_t addr_cluster, uint32_t v) {
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(addr_cluster), "r"(v) : "memory");
}

// TMA load into this CTA's shared memory that signals an mbarrier of either
// CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm, int x, int y,
                                                 uint32_t bar_cluster) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(x), "r"(y), "r"(bar_cluster)
        : "memory");
}

__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
                 "r"(ncols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}

__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}

// Pair MMA (issued by the even CTA): A rows split between the two CTAs (each
// its own shared memory, M/2 rows), B columns split likewise (N/2 each), D
// rows in each CTA's own TMEM.
__device__ __forceinline__ void tc_mma_bf16_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                                 uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Arrive once on the mbarrier at the same offset in every CTA of cta_mask when
// the pair MMAs issued so far have completed.
__device__ __forceinline__ void tc_commit_pair_mc(uint32_t bar, uint16_t cta_mask) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
        "h"(cta_mask)
        : "memory");
}

// 32 lanes x 32 consecutive 32-bit columns from TMEM into registers.
__device__ __forceinline__ void tmem_ld_32x32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor: K-major operand tile written by TMA with
// 128-byte swizzle (rows of 64 bf16, 8-row atoms 1024 bytes apart).
__device__ __forceinline__ uint64_t smem_desc_sw128(uint32_t addr) {
    uint64_t desc = 0;
    desc |= (uint64_t)((addr & 0x3FFFFu) >> 4);        // start address
    desc |= (uint64_t)(16u >> 4) << 16;                 // leading byte offset (unused here)
    desc |= (uint64_t)(1024u >> 4) << 32;               // stride byte offset: 8 rows
    desc |= (uint64_t)1 << 46;                          // descriptor version
    desc |= (uint64_t)2 << 61;                          // 128-byte swizzle
    return desc;
}

// Instruction descriptor, kind::f16: bf16 A and B (K-major), fp32 D, M x N.
__host__ __device__ constexpr uint32_t idesc_bf16_f32(int M, int N) {
    return (1u << 4)                       // D format f32
           | (1u << 7)                     // A format bf16
           | (1u << 10)                    // B format bf16
           | ((uint32_t)(N >> 3) << 17)    // N / 8
           | ((uint32_t)(M >> 4) << 24);   // M / 16
}

__device__ __forceinline__ float bf16_lo(uint32_t v) { return __uint_as_float(v << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t v) { return __uint_as_float(v & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t*>(&v);
}

// cp.async (16 bytes, zero-filled past src_bytes), ldmatrix and mma.sync
// fragments (router and attention kernels).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src, int src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x2(uint32_t (&r)[2], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
                 : "=r"(r[0]), "=r"(r[1])
                 : "r"(addr));
}
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], const uint32_t (&a)[4], const uint32_t (&b)[2]) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
__device__ __forceinline__ void ldmatrix_x4_trans(uint32_t (&r)[4], uint32_t addr) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr));
}

}  // namespace tmoe
