// Host runtime of the C ABI declared in include/trimmoe.h: validation, the
// candidate lists V_{l,r} with their losses Q (Eq. 3), workspaces, TMA
// descriptors, and the per-layer launch sequence
//   decide -> compact -> gather -> FFN gate/up -> FFN down -> combine
// (the per-layer body of Algorithm 2 plus the MoE computation it gates).
#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <limits>
#include <mutex>
#include <string>
#include <utility>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "internal.cuh"

using namespace tmoe;

namespace {

std::mutex g_err_mu;
std::string g_create_error;

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2-D bf16 tensor [outer][inner] with a box of box_outer rows x 64 columns, 128B swizzle.
bool make_tmap(CUtensorMap* tm, const void* base, uint64_t inner, uint64_t outer, uint32_t box_outer) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {inner * 2};
    cuuint32_t box[2] = {64, box_outer};
    cuuint32_t es[2] = {1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box, es,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Small batches: routed GEMMs with at most kSplitKRows executed pairs may split K.
constexpr int kSplitKMax = 8, kSplitKRows = 64;
// GEMM launches whose groups average at least kPairMinRows rows run on CTA
// pairs (256-row tiles): below that the extra padding of a 256-row tail tile
// outweighs the pair's faster main loop.
constexpr int kPairMinRows = 2048;

inline bool pair_gemm(long long rows_per_group) { return rows_per_group >= kPairMinRows; }

// Routed launches whose groups average at least this many rows run their
// store / ReLU epilogues on the transposed pair kernel; smaller groups are
// weight-streaming bound, and its 256-feature pair tiles would leave a ragged
// last round (Mixtral-shaped decode at 256 tokens: 15.2 -> 15.6 ms per step).
constexpr int kTransposedMinRows = 256;

// CTA-pair launches with at least this K draw their tiles from a launch-wide
// counter (a pair whose tiles ran short takes more of them); at shorter K the
// per-tile hand-off costs more than the balance saves (transposed launches:
// Switch-shaped forward 1.011 -> 1.034 ms, Mixtral-shaped 198.3 -> 196.5 ms).
constexpr int kDynamicMinK = 4096;

inline bool dynamic_tiles(int K) { return K >= kDynamicMinK; }

// Tile counters per layer, one per CTA-pair launch: routed up, routed down,
// shared up, shared down, q/k/v projection, output projection.
enum SchedSlot { SCHED_UP = 0, SCHED_DOWN, SCHED_SH_UP, SCHED_SH_DOWN, SCHED_QKV, SCHED_O, SCHED_SLOTS };

enum Kind { K_DECIDE = 0, K_COMPACT, K_GATHER, K_GEMM_UP, K_GEMM_DOWN, K_COMBINE, K_ROUTER, K_ATTN, K_ATTN_GEMM, K_NUM };

// NVTX range names per kernel family, nested in "trimmoe.layer_step" (itself
// inside "trimmoe.forward" for a forward): a profiler can select a family's
// kernels by the host ranges they were launched in, e.g. ncu --nvtx
// --nvtx-include "trimmoe.layer_step/gemm_down/".  Host-side markers only: a
// replayed forward graph is launched by one call, so its kernels carry only
// the range open at that call ("trimmoe.forward").
const char* const kKindName[K_NUM] = {"decide", "compact", "gather", "gemm_up", "gemm_down",
                                      "combine", "router", "attn", "attn_gemm"};

struct NvtxRange {
    explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange&) = delete;
    NvtxRange& operator=(const NvtxRange&) = delete;
};

inline float bf16_to_float(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    std::memcpy(&f, &u, 4);
    return f;
}

inline uint16_t float_to_bf16(float f) {   // round to nearest even (finite inputs)
    uint32_t u;
    std::memcpy(&u, &f, 4);
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

struct DeviceGuard {
    int prev = -1;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) cudaSetDevice(dev);
        else prev = -1;
    }
    ~DeviceGuard() {
        if (prev >= 0) cudaSetDevice(prev);
    }
};

}  // namespace

void tmoe::set_global_error(const std::string& msg) {
    std::lock_guard<std::mutex> g(g_err_mu);
    g_create_error = msg;
}

// A captured forward (all layers) replayed as one CUDA graph.  Two instances
// alternate so that the profiling events of one replay can be read while the
// next one runs.
struct GraphInst {
    cudaGraphExec_t exec = nullptr;
    std::vector<std::pair<std::pair<cudaEvent_t, cudaEvent_t>, int>> evs;   // profile events inside the graph
    bool pending = false;                                                   // replay not read yet
};

struct ForwardGraph {
    int T = -1;
    trimmoe_tokens tok = {};
    cudaStream_t st = nullptr;
    int eager_runs = 0;          // forwards run eagerly with this key (the first one is)
    GraphInst inst[2];
    int next = 0;
    // host-side counters one replay adds
    uint64_t launches = 0, layer_calls = 0, n_gemm_up = 0, n_gemm_down = 0;
    double flops_attn = 0.0, flops_attn_gemm = 0.0;
};

struct trimmoe {
    trimmoe_config cfg;
    trimmoe_weights w;
    int dev = 0, num_sms = 0, n13 = 1;
    std::string err;
    cudaStream_t last_stream = nullptr;
    std::vector<void*> allocs;

    // decision tables
    uint8_t* cand_m = nullptr;
    uint8_t* cand_k = nullptr;
    float* cand_Q = nullptr;
    int* cand_off = nullptr;
    __nv_bfloat16* rt_hi = nullptr;   // [N][E+C][d] router (gamma folded, hi part) then exit head of layer-1
    __nv_bfloat16* rt_lo = nullptr;   // [N][E][d] lo part of gamma * W_r
    float* rt_bias = nullptr;         // [N][E+C]
    // Shared look-ahead tables: per layer the sorted distinct thresholds (Q of
    // the candidates and eps of the window's layers), the depths tabulated and
    // the table workspace of the current layer.
    std::vector<float> h_thr;         // flat, layer after layer
    std::vector<int> thr_off;         // [N + 1]
    std::vector<int> tab_depths;      // [N] depths tabulated (0: none)
    float* thr = nullptr;
    float* phi_tabs = nullptr;
    // Every layer's tables in one buffer (la_all): layer l's at tab_off, built
    // by one launch at the start of a forward (tabs_ready while its layers run).
    bool la_all = false, tabs_ready = false;
    std::vector<LaLayer> h_la;
    LaLayer* la_layers = nullptr;
    int la_max_thr = 0, la_max_depth = 0;
    float* dbar_shared = nullptr;     // [1]
    float* cnorm = nullptr;           // [N][K_c] centroid norms
    int16_t* lhat = nullptr;          // [N][K_c] rounded average exit layers
    float* zbuf = nullptr;            // [rows_part][E+C+K_c] partial logits
    float* sqbuf = nullptr;           // [rows_part] partial sums of squares
    size_t rows_part = 0;             // max over T <= T_max of ksplit(T) * T
    float* ctab = nullptr;
    int max_layer_cand = 1;
    float *trans = nullptr, *comp = nullptr, *P = nullptr, *theta = nullptr, *lambda = nullptr, *eps = nullptr;

    // workspaces
    int32_t* topk_idx = nullptr;
    float* topk_g = nullptr;
    float* I = nullptr;
    float* xi = nullptr;
    uint8_t* action = nullptr;
    uint8_t* exp_sel = nullptr;
    uint8_t* srv_sel = nullptr;
    int32_t *perm = nullptr, *pos_pair = nullptr, *pos_sh = nullptr, *goff = nullptr;
    float* rnorm = nullptr;
    int32_t* blk_counts = nullptr;
    __nv_bfloat16 *Xp = nullptr, *act = nullptr, *act_sh = nullptr, *Y = nullptr, *Ysh = nullptr;
    DevCounters* ctr = nullptr;
    int* dev_err = nullptr;
    float* splitk = nullptr;          // [8][64][max(n13 F, d)] partial sums of split-K GEMMs
    int* gemm_sched = nullptr;        // [N][SCHED_SLOTS] tile counters of a layer's CTA-pair GEMM launches
    bool sched_any = false;           // some launch draws its tiles from a counter
    // Counter of a layer's launch of depth K, or null (static tile order).
    int* sched_for(int layer, int slot, int K) const {
        return dynamic_tiles(K) ? gemm_sched + (size_t)layer * SCHED_SLOTS + slot : nullptr;
    }
    float* la_scratch = nullptr;      // per-token look-ahead scratch of the decision kernel (shared-table layers)
    // Side stream for the shared look-ahead tables: they depend only on the
    // tables and the budget, so they are computed while the router runs.
    cudaStream_t aux = nullptr;
    cudaEvent_t ev_fork = nullptr, ev_join = nullptr;
    int rows_xp = 0;

    CUtensorMap tmXp, tmAct, tmActSh;
    std::vector<CUtensorMap> tmW13, tmW2, tmW13sh, tmW2sh;
    // the same weights in 128-row boxes (each CTA's half of a B tile in the pair kernel)
    std::vector<CUtensorMap> tmW13p, tmW2p, tmW13shp, tmW2shp;

    // attention sublayer of the full block
    int nqkv = 0;
    __nv_bfloat16 *qkv = nullptr, *attn_out = nullptr, *hm = nullptr;
    // Value heads transposed per sequence [seq][Hkv * Dh][kVtSlots] (keys
    // contiguous: the K-major operand of O = P V), zeroed at create.
    __nv_bfloat16* vt = nullptr;
    size_t vt_elems = 0;
    int* goff_attn = nullptr;
    float2* rope = nullptr;           // [attn_seq][head_dim/2] (cos, sin)
    float* sqbuf_x = nullptr;         // [rows_part] partial sums of squares of the layer input
    CUtensorMap tmAttn;
    std::vector<CUtensorMap> tmWqkv, tmWo, tmWqkvp, tmWop;
    // router weight rows per layer (64-column boxes): hi and lo of the router
    // pass, and the exit-head / centroid rows read from the layer input (full block)
    std::vector<CUtensorMap> tmRhi, tmRlo, tmRxhi;
    double flops_attn = 0.0, flops_attn_gemm = 0.0;

    // host-buffer forward
    trimmoe_tokens dtok = {};

    // runtime feedback: host copies of the delay tables, window counters, scratch
    std::vector<float> h_trans, h_comp;
    double win_delay0 = 0.0, win_ref_slots = 0.0;
    double* fb_util = nullptr;
    int* fb_updated = nullptr;
    double* fb_result = nullptr;

    // offline-stage calibration counts
    int calib = 0;
    int16_t* prev_target = nullptr;
    unsigned long long* c_counts = nullptr;   // trans | alive | resid | act | above
    size_t n_counts = 0;

    // counters kept on the host
    uint64_t launches = 0, layer_calls = 0;

    // CUDA graph of the forward (cfg.graphs), and the event list a capture fills
    ForwardGraph fg;
    std::vector<std::pair<std::pair<cudaEvent_t, cudaEvent_t>, int>>* cap_evs = nullptr;

    // profiling
    std::vector<cudaEvent_t> ev_free;
    std::vector<std::pair<std::pair<cudaEvent_t, cudaEvent_t>, int>> ev_pending;
    double ms[K_NUM] = {0};
    uint64_t n_gemm_up = 0, n_gemm_down = 0;

    trimmoe_status fail(trimmoe_status s, const std::string& m) {
        err = m;
        return s;
    }

    template <class T>
    bool dalloc(T** p, size_t n) {
        void* q = nullptr;
        if (n == 0) n = 1;
        if (cudaMalloc(&q, n * sizeof(T)) != cudaSuccess) {
            cudaGetLastError();
            return false;
        }
        allocs.push_back(q);
        *p = static_cast<T*>(q);
        return true;
    }

    cudaEvent_t get_event() {
        if (!ev_free.empty()) {
            cudaEvent_t e = ev_free.back();
            ev_free.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        cudaEventCreate(&e);
        return e;
    }

    // Launch helper: records profile events around fn() when enabled.
    template <class Fn>
    cudaError_t timed(int kind, cudaStream_t st, Fn fn) {
        NvtxRange range(kKindName[kind]);
        cudaEvent_t a = nullptr, b = nullptr;
        // Inside a stream capture the events become event-record nodes of the
        // graph (cudaEventRecordExternal), recorded at every replay.
        const unsigned rec_flags = cap_evs ? cudaEventRecordExternal : 0u;
        const bool rec = cfg.profile == 1 ||
                         (cfg.profile == 2 && (kind == K_GEMM_UP || kind == K_GEMM_DOWN || kind == K_ATTN_GEMM));
        if (rec) {
            a = get_event();
            b = get_event();
            cudaEventRecordWithFlags(a, st, rec_flags);
        }
        cudaError_t e = fn();
        if (rec) {
            cudaEventRecordWithFlags(b, st, rec_flags);
            (cap_evs ? *cap_evs : ev_pending).push_back({{a, b}, kind});
        }
        return e;
    }

    // Adds the kernel times of a finished graph replay (waits for it if needed).
    void read_graph_inst(GraphInst& gi) {
        if (!gi.pending) return;
        if (!gi.evs.empty()) cudaEventSynchronize(gi.evs.back().first.second);
        for (auto& pe : gi.evs) {
            float t = 0.f;
            if (cudaEventElapsedTime(&t, pe.first.first, pe.first.second) == cudaSuccess) ms[pe.second] += t;
        }
        gi.pending = false;
    }

    void drop_graph() {
        for (GraphInst& gi : fg.inst) {
            read_graph_inst(gi);
            if (gi.exec) cudaGraphExecDestroy(gi.exec);
            gi.exec = nullptr;
            for (auto& pe : gi.evs) {
                ev_free.push_back(pe.first.first);
                ev_free.push_back(pe.first.second);
            }
            gi.evs.clear();
        }
        fg = ForwardGraph();
    }

    void drain_events() {
        for (GraphInst& gi : fg.inst) read_graph_inst(gi);
        for (auto& pe : ev_pending) {
            float t = 0.f;
            if (cudaEventElapsedTime(&t, pe.first.first, pe.first.second) == cudaSuccess) ms[pe.second] += t;
            ev_free.push_back(pe.first.first);
            ev_free.push_back(pe.first.second);
        }
        ev_pending.clear();
    }
};

namespace {

// Delay part of the execute cost, omega_T * (d(m -> m') / d_ref) with
// d(m -> m') = trans[m][m'] (m != m') + comp[l][m'] (Eq. 30-31), in fp32.
std::vector<float> delay_cost_table(const trimmoe_config& c, const std::vector<float>& trans,
                                    const std::vector<float>& comp) {
    const int N = c.N, M = c.M;
    std::vector<float> ctab((size_t)N * M * M);
    for (int l = 0; l < N; ++l)
        for (int m = 0; m < M; ++m)
            for (int mp = 0; mp < M; ++mp) {
                const float tr = (mp != m) ? trans[(size_t)m * M + mp] : 0.0f;
                const float dly = tr + comp[(size_t)l * M + mp];
                ctab[((size_t)l * M + m) * M + mp] = c.omega_T * (dly / c.d_ref_ms);
            }
    return ctab;
}

trimmoe_status validate_config(const trimmoe_config* c, std::string& why) {
    if (c->N < 1 || c->d < 1 || c->E < 1 || c->k < 1 || c->F < 1 || c->M < 1 || c->H < 1 || c->C < 1 ||
        c->T_max < 1 || c->F_sh < 0 || c->n_sub < 0) {
        why = "config: every dimension must be positive";
        return TRIMMOE_ERR_ARG;
    }
    if (c->act != 0 && c->act != 1) { why = "config: act must be 0 (ReLU) or 1 (SwiGLU)"; return TRIMMOE_ERR_ARG; }
    if (!(c->d_ref_ms > 0.f) || !std::isfinite(c->d_ref_ms)) { why = "config: d_ref_ms must be > 0"; return TRIMMOE_ERR_ARG; }
    if (!(c->norm_eps >= 0.f) || !std::isfinite(c->norm_eps)) { why = "config: norm_eps must be >= 0"; return TRIMMOE_ERR_ARG; }
    if (c->d % 256) { why = "config: d must be a multiple of 256"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->d > 16384) { why = "config: d > 16384"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->act == 1 && c->F % 128) { why = "config: SwiGLU F must be a multiple of 128"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->act == 0 && c->F % 256) { why = "config: ReLU F must be a multiple of 256"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->F_sh % 128) { why = "config: F_sh must be a multiple of 128"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->E > kMaxE) { why = "config: E > 128"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->k > kMaxK || c->k > c->E) { why = "config: k must be <= min(E, 8)"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->M > kMaxM) { why = "config: M > 16"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->C > kMaxC) { why = "config: C > 256"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->M * c->E > kMaxME) { why = "config: M*E > 1024"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->H > kMaxH) { why = "config: H > 6"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->n_sub > 3) { why = "config: n_sub > 3"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->n_centroids < 0 || c->n_centroids > 256) { why = "config: n_centroids must be in [0, 256]"; return TRIMMOE_ERR_UNSUPPORTED; }
    if ((long long)c->T_max * (c->k + 1) >= (1ll << 31)) { why = "config: T_max too large"; return TRIMMOE_ERR_UNSUPPORTED; }
    if (c->profile < 0 || c->profile > 2) { why = "config: profile must be 0, 1 or 2"; return TRIMMOE_ERR_ARG; }
    if (c->graphs != 0 && c->graphs != 1) { why = "config: graphs must be 0 or 1"; return TRIMMOE_ERR_ARG; }
    if (c->attn_heads < 0) { why = "config: attn_heads must be >= 0"; return TRIMMOE_ERR_ARG; }
    if (c->attn_heads > 0) {
        if (c->attn_kv_heads < 1 || c->attn_heads % c->attn_kv_heads) {
            why = "config: attn_heads must be a positive multiple of attn_kv_heads";
            return TRIMMOE_ERR_ARG;
        }
        if (c->head_dim != 64 && c->head_dim != 128) { why = "config: head_dim must be 64 or 128"; return TRIMMOE_ERR_UNSUPPORTED; }
        if (((long long)c->attn_heads + 2 * c->attn_kv_heads) * c->head_dim % 256) {
            why = "config: (attn_heads + 2 attn_kv_heads) * head_dim must be a multiple of 256";
            return TRIMMOE_ERR_UNSUPPORTED;
        }
        if (c->attn_seq < 1 || c->attn_seq > 128) { why = "config: attn_seq must be in [1, 128]"; return TRIMMOE_ERR_UNSUPPORTED; }
        if (!(c->rope_theta > 1.f) || !std::isfinite(c->rope_theta)) { why = "config: rope_theta must be > 1"; return TRIMMOE_ERR_ARG; }
    }
    return TRIMMOE_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace

extern "C" trimmoe_status trimmoe_create(const trimmoe_config* cfg, const trimmoe_weights* w,
                                         const trimmoe_tables* tab, trimmoe_handle* out) {
    auto create_fail = [&](trimmoe_status s, const std::string& m) {
        std::lock_guard<std::mutex> g(g_err_mu);
        g_create_error = m;
        return s;
    };
    if (!out) return create_fail(TRIMMOE_ERR_ARG, "create: out is NULL");
    *out = nullptr;
    if (!cfg || !w || !tab) return create_fail(TRIMMOE_ERR_ARG, "create: NULL argument");
    std::string why;
    trimmoe_status st = validate_config(cfg, why);
    if (st != TRIMMOE_OK) return create_fail(st, why);
    const trimmoe_config c = *cfg;
    const int N = c.N, E = c.E, M = c.M, d = c.d;
    const int n13 = c.act == 1 ? 2 : 1;
    if (!w->W_r || !w->b_r || !w->W_x || !w->b_x || !w->W13 || !w->W2)
        return create_fail(TRIMMOE_ERR_ARG, "create: NULL weight pointer");
    if (c.n_centroids > 0 && (!w->centroids || !tab->centroid_exit || !aligned16(w->centroids)))
        return create_fail(TRIMMOE_ERR_ARG, "create: n_centroids > 0 needs 16-byte aligned centroids and centroid_exit");
    if (c.attn_heads > 0 && (!w->W_attn_norm || !w->W_qkv || !w->W_o || !w->W_norm))
        return create_fail(TRIMMOE_ERR_ARG, "create: the attention sublayer needs W_attn_norm, W_qkv, W_o and W_norm");
    if (c.attn_heads > 0 && (!aligned16(w->W_attn_norm) || !aligned16(w->W_qkv) || !aligned16(w->W_o)))
        return create_fail(TRIMMOE_ERR_ARG, "create: weights must be 16-byte aligned");
    if ((c.F_sh > 0) != (w->W13_sh != nullptr && w->W2_sh != nullptr))
        return create_fail(TRIMMOE_ERR_ARG, "create: shared-expert weights must be given iff F_sh > 0");
    if (!aligned16(w->W_r) || !aligned16(w->W_x) || !aligned16(w->W13) || !aligned16(w->W2) ||
        (c.F_sh && (!aligned16(w->W13_sh) || !aligned16(w->W2_sh))) || (w->W_norm && !aligned16(w->W_norm)))
        return create_fail(TRIMMOE_ERR_ARG, "create: weights must be 16-byte aligned");
    if (!tab->place || !tab->sim || !tab->sub_thresh || !tab->trans_ms || !tab->comp_ms || !tab->theta ||
        !tab->lambda || !tab->eps || (N > 1 && !tab->P))
        return create_fail(TRIMMOE_ERR_ARG, "create: NULL table pointer");

    // Coverage (Eq. 2) and table sanity.
    const uint32_t mmask = (M >= 16) ? 0xFFFFu : ((1u << M) - 1u);
    for (int l = 0; l < N; ++l)
        for (int e = 0; e < E; ++e)
            if ((tab->place[l * E + e] & mmask) == 0) {
                char b[96];
                snprintf(b, sizeof b, "create: expert %d of layer %d has no server (Eq. 2)", e, l);
                return create_fail(TRIMMOE_ERR_COVERAGE, b);
            }
    for (int i = 0; i < M * M; ++i)
        if (!(tab->trans_ms[i] >= 0.f) || !std::isfinite(tab->trans_ms[i]))
            return create_fail(TRIMMOE_ERR_ARG, "create: trans_ms must be finite and >= 0");
    for (int i = 0; i < N * M; ++i)
        if (!(tab->comp_ms[i] >= 0.f) || !std::isfinite(tab->comp_ms[i]))
            return create_fail(TRIMMOE_ERR_ARG, "create: comp_ms must be finite and >= 0");
    for (int l = 0; l + 1 < N; ++l)
        for (int k = 0; k < E; ++k) {
            double s = 0;
            for (int kp = 0; kp < E; ++kp) {
                const float v = tab->P[((size_t)l * E + k) * E + kp];
                if (!(v >= 0.f) || !std::isfinite(v)) return create_fail(TRIMMOE_ERR_ARG, "create: P entries must be >= 0");
                s += v;
            }
            if (std::fabs(s - 1.0) > 1e-3) return create_fail(TRIMMOE_ERR_ARG, "create: P rows must sum to 1");
        }

    trimmoe* h = new (std::nothrow) trimmoe();
    if (!h) return create_fail(TRIMMOE_ERR_OOM, "create: host allocation failed");
    h->cfg = c;
    h->w = *w;
    h->n13 = n13;
    auto bail = [&](trimmoe_status s, const std::string& m) {
        trimmoe_destroy(h);
        return create_fail(s, m);
    };
    if (cudaGetDevice(&h->dev) != cudaSuccess) return bail(TRIMMOE_ERR_CUDA, "create: no CUDA device");
    cudaDeviceProp prop;
    if (cudaGetDeviceProperties(&prop, h->dev) != cudaSuccess) return bail(TRIMMOE_ERR_CUDA, "create: device query failed");
    if (prop.major != 10) return bail(TRIMMOE_ERR_UNSUPPORTED, "create: needs a Blackwell (sm_10x) device");
    h->num_sms = prop.multiProcessorCount;

    // Candidate lists V_{l,r} (Sec. III-A): the exact expert, then the n_sub
    // most similar experts with Sim >= sub_thresh (ties to the lower index),
    // by expert index; servers ascending within an expert (Eq. 11).  Stored
    // flat, layer after layer, with per-(layer, target) offsets.
    std::vector<uint8_t> cm, ck;
    std::vector<float> cq;
    std::vector<int> coff((size_t)N * (E + 1), 0);
    int max_layer_cand = 1;
    for (int l = 0; l < N; ++l) {
        const int layer_start = (int)cm.size();
        for (int r = 0; r < E; ++r) {
            coff[(size_t)l * (E + 1) + r] = (int)cm.size();
            const float* srow = tab->sim + ((size_t)l * E + r) * E;
            std::vector<std::pair<float, int>> el;
            for (int k = 0; k < E; ++k)
                if (k != r && srow[k] >= tab->sub_thresh[l]) el.push_back({srow[k], k});
            std::sort(el.begin(), el.end(), [](const std::pair<float, int>& a, const std::pair<float, int>& b) {
                return a.first > b.first || (a.first == b.first && a.second < b.second);
            });
            std::vector<int> ex;
            for (size_t i = 0; i < el.size() && (int)i < c.n_sub; ++i) ex.push_back(el[i].second);
            std::sort(ex.begin(), ex.end());
            ex.insert(ex.begin(), r);
            for (int k : ex) {
                const float q = (k == r) ? 0.0f : c.phi_beta * ((1.0f - srow[k]) / 2.0f);
                for (int m = 0; m < M; ++m)
                    if ((tab->place[l * E + k] >> m) & 1u) {
                        cm.push_back((uint8_t)m);
                        ck.push_back((uint8_t)k);
                        cq.push_back(q);
                    }
            }
        }
        coff[(size_t)l * (E + 1) + E] = (int)cm.size();
        max_layer_cand = std::max(max_layer_cand, (int)cm.size() - layer_start);
    }
    h->h_trans.assign(tab->trans_ms, tab->trans_ms + (size_t)M * M);
    h->h_comp.assign(tab->comp_ms, tab->comp_ms + (size_t)N * M);
    std::vector<float> ctab = delay_cost_table(c, h->h_trans, h->h_comp);
    if (decide_smem_bytes(E, c.C, M, max_layer_cand) > 200 * 1024) {
        trimmoe_destroy(h);
        return create_fail(TRIMMOE_ERR_UNSUPPORTED, "create: candidate lists too long for the decision kernel");
    }
    h->max_layer_cand = max_layer_cand;
    // Look-ahead thresholds (Eq. 39): Phi of layer l depends on R only through
    // Q <= R and eps <= R over layers l+1 .. l+top, so the sorted distinct
    // values split R into intervals of equal tables.  Depths below the full
    // window are tabulated only when exit prediction can shorten it.
    h->thr_off.assign(N + 1, 0);
    h->tab_depths.assign(N, 0);
    size_t tab_floats = 0;
    for (int l = 0; l < N; ++l) {
        const int top = std::min(c.H - 1, N - 1 - l);
        std::vector<float> v;
        for (int j = 1; j <= top; ++j) {
            const int lp = l + j;
            v.push_back(tab->eps[lp]);
            for (int i = coff[(size_t)lp * (E + 1)]; i < coff[(size_t)lp * (E + 1) + E]; ++i) v.push_back(cq[i]);
        }
        std::sort(v.begin(), v.end());
        v.erase(std::unique(v.begin(), v.end()), v.end());
        const int depths = top <= 0 ? 0 : (c.n_centroids > 0 ? top : 1);
        const size_t need = (size_t)depths * (v.size() + 1) * M * E;
        if (v.size() + 1 <= kMaxIntervals && need <= kMaxTabFloats) {
            h->tab_depths[l] = depths;
            tab_floats = std::max(tab_floats, need);
        }
        h->h_thr.insert(h->h_thr.end(), v.begin(), v.end());
        h->thr_off[l + 1] = (int)h->h_thr.size();
    }
    // All layers' tables side by side when they fit in kMaxAllTabFloats.
    {
        size_t total = 0;
        h->h_la.assign(N, LaLayer{0, 0, 0, 0});
        for (int l = 0; l < N; ++l) {
            LaLayer& L = h->h_la[l];
            L.thr_off = h->thr_off[l];
            L.n_thr = h->thr_off[l + 1] - h->thr_off[l];
            L.n_depth = h->tab_depths[l];
            L.tab_off = (int)total;
            total += (size_t)L.n_depth * (L.n_thr + 1) * M * E;
            if (L.n_depth > 0) {
                h->la_max_thr = std::max(h->la_max_thr, L.n_thr);
                h->la_max_depth = std::max(h->la_max_depth, L.n_depth);
            }
        }
        h->la_all = total > 0 && total <= kMaxAllTabFloats;
        if (h->la_all) tab_floats = total;
    }

    // Router tables of kernel a0 (built from the borrowed device weights): per
    // layer, rows [0, E) hold gamma_l * W_r[l] split exactly into bf16 hi + lo
    // (a bf16 x bf16 product has at most 16 significant bits), rows [E, E+C) the
    // exit head of layer l-1 (zero at layer 0); biases likewise.
    const int Kc = c.n_centroids;
    const int n_out = E + c.C + Kc;
    std::vector<uint16_t> hWr((size_t)N * E * d), hWx((size_t)N * c.C * d), hG, hCt((size_t)N * Kc * d);
    std::vector<float> hbr((size_t)N * E), hbx((size_t)N * c.C);
    {
        cudaError_t e1 = cudaMemcpy(hWr.data(), w->W_r, hWr.size() * 2, cudaMemcpyDeviceToHost);
        if (e1 == cudaSuccess) e1 = cudaMemcpy(hWx.data(), w->W_x, hWx.size() * 2, cudaMemcpyDeviceToHost);
        if (e1 == cudaSuccess) e1 = cudaMemcpy(hbr.data(), w->b_r, hbr.size() * 4, cudaMemcpyDeviceToHost);
        if (e1 == cudaSuccess) e1 = cudaMemcpy(hbx.data(), w->b_x, hbx.size() * 4, cudaMemcpyDeviceToHost);
        if (e1 == cudaSuccess && w->W_norm) {
            hG.resize((size_t)N * d);
            e1 = cudaMemcpy(hG.data(), w->W_norm, hG.size() * 2, cudaMemcpyDeviceToHost);
        }
        if (e1 == cudaSuccess && Kc > 0)
            e1 = cudaMemcpy(hCt.data(), w->centroids, hCt.size() * 2, cudaMemcpyDeviceToHost);
        if (e1 != cudaSuccess) return bail(TRIMMOE_ERR_CUDA, std::string("create: reading router weights: ") + cudaGetErrorString(e1));
    }
    std::vector<uint16_t> rhi((size_t)N * n_out * d, 0), rlo((size_t)N * E * d, 0);
    std::vector<float> rb((size_t)N * n_out, 0.f);
    for (int l = 0; l < N; ++l) {
        for (int e = 0; e < E; ++e) {
            for (int i = 0; i < d; ++i) {
                const float wv = bf16_to_float(hWr[((size_t)l * E + e) * d + i]);
                const float prod = hG.empty() ? wv : wv * bf16_to_float(hG[(size_t)l * d + i]);
                const uint16_t hi = float_to_bf16(prod);
                const uint16_t lo = float_to_bf16(prod - bf16_to_float(hi));
                rhi[((size_t)l * n_out + e) * d + i] = hi;
                rlo[((size_t)l * E + e) * d + i] = lo;
            }
            rb[(size_t)l * n_out + e] = hbr[(size_t)l * E + e];
        }
        if (l > 0)
            for (int cc = 0; cc < c.C; ++cc) {
                std::memcpy(&rhi[((size_t)l * n_out + E + cc) * d], &hWx[((size_t)(l - 1) * c.C + cc) * d], (size_t)d * 2);
                rb[(size_t)l * n_out + E + cc] = hbx[(size_t)(l - 1) * c.C + cc];
            }
        for (int j = 0; j < Kc; ++j)
            std::memcpy(&rhi[((size_t)l * n_out + E + c.C + j) * d], &hCt[((size_t)l * Kc + j) * d], (size_t)d * 2);
    }
    // Centroid norms (double sum, rounded to fp32) and rounded exit layers (Eq. 36).
    std::vector<float> cn((size_t)N * std::max(Kc, 1), 0.f);
    std::vector<int16_t> lh((size_t)N * std::max(Kc, 1), 0);
    for (int l = 0; l < N; ++l)
        for (int j = 0; j < Kc; ++j) {
            double nn = 0.0;
            for (int i = 0; i < d; ++i) {
                const double v = bf16_to_float(hCt[((size_t)l * Kc + j) * d + i]);
                nn += v * v;
            }
            cn[(size_t)l * Kc + j] = (float)std::sqrt(nn);
            lh[(size_t)l * Kc + j] = (int16_t)std::floor((double)tab->centroid_exit[(size_t)l * Kc + j] + 0.5);
        }

    for (int tt = 1; tt <= c.T_max; ++tt)
        h->rows_part = std::max(h->rows_part, (size_t)router_ksplit(tt, d, n_out, h->num_sms) * tt);

    // Device tables and workspaces.
    const size_t T = (size_t)c.T_max, TK = T * c.k;
    const int has_sh = c.F_sh > 0;
    h->rows_xp = (int)(TK + (has_sh ? T : 0));
    const int nblk = (int)((T + 255) / 256);
    bool ok = h->dalloc(&h->cand_m, cm.size()) && h->dalloc(&h->cand_k, ck.size()) &&
              h->dalloc(&h->cand_Q, cq.size()) && h->dalloc(&h->cand_off, coff.size()) &&
              h->dalloc(&h->ctab, ctab.size()) && h->dalloc(&h->rt_hi, rhi.size()) &&
              h->dalloc(&h->rt_lo, rlo.size()) && h->dalloc(&h->rt_bias, rb.size()) &&
              h->dalloc(&h->cnorm, cn.size()) && h->dalloc(&h->lhat, lh.size()) &&
              h->dalloc(&h->zbuf, h->rows_part * (size_t)n_out) && h->dalloc(&h->sqbuf, h->rows_part) &&
              h->dalloc(&h->trans, (size_t)M * M) && h->dalloc(&h->comp, (size_t)N * M) &&
              h->dalloc(&h->P, (size_t)std::max(N - 1, 1) * E * E) && h->dalloc(&h->theta, N) &&
              h->dalloc(&h->lambda, N) && h->dalloc(&h->eps, N) && h->dalloc(&h->topk_idx, TK) &&
              h->dalloc(&h->topk_g, TK) && h->dalloc(&h->I, T) && h->dalloc(&h->xi, T) &&
              h->dalloc(&h->action, T) && h->dalloc(&h->exp_sel, TK) && h->dalloc(&h->srv_sel, TK) &&
              h->dalloc(&h->perm, TK + T) && h->dalloc(&h->pos_pair, TK) && h->dalloc(&h->pos_sh, T) &&
              h->dalloc(&h->rnorm, T) &&
              h->dalloc(&h->goff, (size_t)E + 2) && h->dalloc(&h->blk_counts, (size_t)nblk * (E + 1)) &&
              h->dalloc(&h->Xp, (size_t)h->rows_xp * d) && h->dalloc(&h->act, TK * c.F) &&
              h->dalloc(&h->Y, TK * d) && h->dalloc(&h->ctr, kCtrCopies) && h->dalloc(&h->dev_err, 1) &&
              h->dalloc(&h->fb_util, T) && h->dalloc(&h->fb_updated, T) && h->dalloc(&h->fb_result, 2) &&
              h->dalloc(&h->prev_target, T) && h->dalloc(&h->phi_tabs, std::max<size_t>(tab_floats, 1)) &&
              h->dalloc(&h->thr, std::max<size_t>(h->h_thr.size(), 1)) && h->dalloc(&h->dbar_shared, 1) &&
              (!h->la_all || h->dalloc(&h->la_layers, (size_t)N));
    h->n_counts = (size_t)std::max(N - 1, 1) * E * E + N + (size_t)N * M + 2 * (size_t)N * E;
    ok = ok && h->dalloc(&h->c_counts, h->n_counts) &&
         h->dalloc(&h->splitk, (size_t)kSplitKMax * kSplitKRows * std::max<size_t>((size_t)h->n13 * c.F, (size_t)d)) &&
         h->dalloc(&h->gemm_sched, (size_t)SCHED_SLOTS * N);
    if (ok && has_sh) ok = h->dalloc(&h->act_sh, T * c.F_sh) && h->dalloc(&h->Ysh, T * d);
    if (ok && tab_floats > 0)
        ok = h->dalloc(&h->la_scratch, decide_la_scratch_floats(E, M, h->max_layer_cand, h->num_sms));
    const int has_attn = c.attn_heads > 0;
    if (has_attn) {
        h->nqkv = (c.attn_heads + 2 * c.attn_kv_heads) * c.head_dim;
        ok = ok && h->dalloc(&h->qkv, T * h->nqkv) && h->dalloc(&h->attn_out, T * c.attn_heads * c.head_dim) &&
             h->dalloc(&h->hm, T * d) && h->dalloc(&h->goff_attn, 2) &&
             h->dalloc(&h->rope, (size_t)c.attn_seq * (c.head_dim / 2)) && h->dalloc(&h->sqbuf_x, h->rows_part);
        h->vt_elems = ((T + c.attn_seq - 1) / c.attn_seq) * (size_t)c.attn_kv_heads * c.head_dim * kVtSlots;
        ok = ok && h->dalloc(&h->vt, h->vt_elems);
    }
    if (!ok) return bail(TRIMMOE_ERR_OOM, "create: device allocation failed");
    cudaError_t ce = cudaSuccess;
    auto up = [&](void* dst, const void* src, size_t bytes) {
        if (ce == cudaSuccess) ce = cudaMemcpy(dst, src, bytes, cudaMemcpyHostToDevice);
    };
    up(h->cand_m, cm.data(), cm.size());
    up(h->cand_k, ck.data(), ck.size());
    up(h->cand_Q, cq.data(), cq.size() * 4);
    if (!h->h_thr.empty()) up(h->thr, h->h_thr.data(), h->h_thr.size() * 4);
    if (h->la_all) up(h->la_layers, h->h_la.data(), h->h_la.size() * sizeof(LaLayer));
    up(h->cand_off, coff.data(), coff.size() * 4);
    up(h->ctab, ctab.data(), ctab.size() * 4);
    up(h->rt_hi, rhi.data(), rhi.size() * 2);
    up(h->rt_lo, rlo.data(), rlo.size() * 2);
    up(h->rt_bias, rb.data(), rb.size() * 4);
    up(h->cnorm, cn.data(), cn.size() * 4);
    up(h->lhat, lh.data(), lh.size() * 2);
    up(h->trans, tab->trans_ms, (size_t)M * M * 4);
    up(h->comp, tab->comp_ms, (size_t)N * M * 4);
    if (N > 1) up(h->P, tab->P, (size_t)(N - 1) * E * E * 4);
    up(h->theta, tab->theta, N * 4);
    up(h->lambda, tab->lambda, N * 4);
    up(h->eps, tab->eps, N * 4);
    if (has_attn) {
        // Rotary table: angle pos * theta^(-2i/Dh), cos and sin in double, stored fp32.
        const int half = c.head_dim / 2;
        std::vector<float2> rt((size_t)c.attn_seq * half);
        for (int pos = 0; pos < c.attn_seq; ++pos)
            for (int i = 0; i < half; ++i) {
                const double ang = (double)pos * std::pow((double)c.rope_theta, -2.0 * i / c.head_dim);
                rt[(size_t)pos * half + i] = make_float2((float)std::cos(ang), (float)std::sin(ang));
            }
        up(h->rope, rt.data(), rt.size() * sizeof(float2));
        // Key slots past a sequence's end are multiplied by zero probabilities:
        // they must never hold NaN, so the buffer starts at zero.
        if (ce == cudaSuccess) ce = cudaMemset(h->vt, 0, h->vt_elems * sizeof(__nv_bfloat16));
    }
    if (ce == cudaSuccess) ce = cudaStreamCreateWithFlags(&h->aux, cudaStreamNonBlocking);
    if (ce == cudaSuccess) ce = cudaEventCreateWithFlags(&h->ev_fork, cudaEventDisableTiming);
    if (ce == cudaSuccess) ce = cudaEventCreateWithFlags(&h->ev_join, cudaEventDisableTiming);
    if (ce == cudaSuccess) ce = cudaMemset(h->ctr, 0, sizeof(DevCounters) * kCtrCopies);
    if (ce == cudaSuccess) ce = cudaMemset(h->dev_err, 0, sizeof(int));
    if (ce == cudaSuccess) ce = cudaMemset(h->gemm_sched, 0, (size_t)SCHED_SLOTS * N * sizeof(int));
    h->sched_any = dynamic_tiles(d) || dynamic_tiles(c.F) || (has_sh && dynamic_tiles(c.F_sh)) ||
                   (c.attn_heads > 0 && dynamic_tiles(c.attn_heads * c.head_dim));
    if (ce == cudaSuccess) ce = cudaMemset(h->Xp, 0, (size_t)h->rows_xp * d * 2);
    if (ce != cudaSuccess) return bail(TRIMMOE_ERR_CUDA, std::string("create: ") + cudaGetErrorString(ce));

    // TMA descriptors: activations (128-row boxes) and per-layer weights (256-row boxes).
    const size_t F13 = (size_t)n13 * c.F;
    bool tm = make_tmap(&h->tmXp, h->Xp, d, h->rows_xp, 128) && make_tmap(&h->tmAct, h->act, c.F, TK, 128);
    if (has_sh) tm = tm && make_tmap(&h->tmActSh, h->act_sh, c.F_sh, T, 128);
    h->tmW13.resize(N);
    h->tmW2.resize(N);
    h->tmW13p.resize(N);
    h->tmW2p.resize(N);
    if (has_sh) { h->tmW13sh.resize(N); h->tmW2sh.resize(N); h->tmW13shp.resize(N); h->tmW2shp.resize(N); }
    const __nv_bfloat16* W13 = static_cast<const __nv_bfloat16*>(w->W13);
    const __nv_bfloat16* W2 = static_cast<const __nv_bfloat16*>(w->W2);
    for (int l = 0; l < N && tm; ++l) {
        for (uint32_t box : {256u, 128u}) {
            CUtensorMap* m13 = box == 256 ? &h->tmW13[l] : &h->tmW13p[l];
            CUtensorMap* m2 = box == 256 ? &h->tmW2[l] : &h->tmW2p[l];
            tm = tm && make_tmap(m13, W13 + (size_t)l * E * F13 * d, d, (uint64_t)E * F13, box) &&
                 make_tmap(m2, W2 + (size_t)l * E * d * c.F, c.F, (uint64_t)E * d, box);
            if (tm && has_sh) {
                const __nv_bfloat16* W13s = static_cast<const __nv_bfloat16*>(w->W13_sh);
                const __nv_bfloat16* W2s = static_cast<const __nv_bfloat16*>(w->W2_sh);
                tm = make_tmap(box == 256 ? &h->tmW13sh[l] : &h->tmW13shp[l], W13s + (size_t)l * 2 * c.F_sh * d, d,
                               (uint64_t)2 * c.F_sh, box) &&
                     make_tmap(box == 256 ? &h->tmW2sh[l] : &h->tmW2shp[l], W2s + (size_t)l * d * c.F_sh, c.F_sh,
                               (uint64_t)d, box);
            }
        }
    }
    if (tm && has_attn) {
        const int hd = c.attn_heads * c.head_dim;
        const __nv_bfloat16* Wqkv = static_cast<const __nv_bfloat16*>(w->W_qkv);
        const __nv_bfloat16* Wo = static_cast<const __nv_bfloat16*>(w->W_o);
        h->tmWqkv.resize(N);
        h->tmWo.resize(N);
        h->tmWqkvp.resize(N);
        h->tmWop.resize(N);
        tm = make_tmap(&h->tmAttn, h->attn_out, hd, T, 128);
        for (int l = 0; l < N && tm; ++l)
            tm = make_tmap(&h->tmWqkv[l], Wqkv + (size_t)l * h->nqkv * d, d, (uint64_t)h->nqkv, 256) &&
                 make_tmap(&h->tmWo[l], Wo + (size_t)l * d * hd, hd, (uint64_t)d, 256) &&
                 make_tmap(&h->tmWqkvp[l], Wqkv + (size_t)l * h->nqkv * d, d, (uint64_t)h->nqkv, 128) &&
                 make_tmap(&h->tmWop[l], Wo + (size_t)l * d * hd, hd, (uint64_t)d, 128);
    }
    if (tm) {
        // Router weights: with the attention sublayer the router rows and the
        // exit-head / centroid rows are read in separate passes over different
        // inputs, so they get separate maps (boxes of one pass's rows).
        h->tmRhi.resize(N);
        h->tmRlo.resize(N);
        if (has_attn) h->tmRxhi.resize(N);
        const int n_main = has_attn ? E : n_out;
        const int ng = router_pass_rows(n_main);
        const int nl = router_lo_rows(E, ng);
        for (int l = 0; l < N && tm; ++l) {
            tm = make_tmap(&h->tmRhi[l], h->rt_hi + (size_t)l * n_out * d, d, (uint64_t)n_main, (uint32_t)ng) &&
                 make_tmap(&h->tmRlo[l], h->rt_lo + (size_t)l * E * d, d, (uint64_t)E, (uint32_t)nl);
            if (tm && has_attn)
                tm = make_tmap(&h->tmRxhi[l], h->rt_hi + ((size_t)l * n_out + E) * d, d, (uint64_t)(n_out - E),
                               (uint32_t)router_pass_rows(n_out - E));
        }
    }
    if (!tm) return bail(TRIMMOE_ERR_CUDA, "create: cuTensorMapEncodeTiled failed");
    *out = h;
    return TRIMMOE_OK;
}

static trimmoe_status check_tokens(trimmoe_handle h, const trimmoe_tokens* tok) {
    if (!tok || !tok->hidden || !tok->s || !tok->Dhat || !tok->Dbar || !tok->pJ || !tok->alive ||
        !tok->last_exec || !tok->xi_last || !tok->exit_layer)
        return h->fail(TRIMMOE_ERR_ARG, "tokens: NULL pointer");
    if (!aligned16(tok->hidden)) return h->fail(TRIMMOE_ERR_ARG, "tokens: hidden must be 16-byte aligned");
    return TRIMMOE_OK;
}

static trimmoe_status layer_step_impl(trimmoe_handle h, int layer, int T, trimmoe_tokens* tok,
                                      trimmoe_layer_out* out, cudaStream_t st) {
    NvtxRange range("trimmoe.layer_step");
    // Launch errors are read with cudaGetLastError after each launch; clear a
    // non-sticky error left behind by other code in this thread first.
    cudaGetLastError();
    const trimmoe_config& c = h->cfg;
    const int E = c.E, K = c.k, d = c.d;
    const int has_sh = c.F_sh > 0;
    const size_t F13 = (size_t)h->n13 * c.F;

    DecideParams dp;
    dp.layer = layer;
    dp.T = T;
    dp.N = c.N;
    dp.d = d;
    dp.E = E;
    dp.k = K;
    dp.C = c.C;
    dp.M = c.M;
    dp.H = c.H;
    dp.omega_T = c.omega_T;
    dp.omega_D = c.omega_D;
    dp.d_ref = c.d_ref_ms;
    const __nv_bfloat16* hid_in = static_cast<const __nv_bfloat16*>(tok->hidden);
    const __nv_bfloat16* hid = hid_in;     // input of the MoE sublayer
    const __nv_bfloat16* gamma =
        h->w.W_norm ? static_cast<const __nv_bfloat16*>(h->w.W_norm) + (size_t)layer * d : nullptr;
    const int Kc = c.n_centroids;
    const int n_out = E + c.C + Kc;
    cudaError_t e = cudaSuccess;
    const bool has_attn = c.attn_heads > 0;
    if (has_attn) {
        // Attention sublayer (Sec. III-C, attention placement): local, for every
        // live token, in front of the MoE decision.
        const int hd = c.attn_heads * c.head_dim;
        AttnParams ap;
        ap.T = T;
        ap.d = d;
        ap.S = c.attn_seq;
        ap.Hq = c.attn_heads;
        ap.Hkv = c.attn_kv_heads;
        ap.nqkv = h->nqkv;
        ap.norm_eps = c.norm_eps;
        ap.scale = (float)(1.0 / std::sqrt((double)c.head_dim));
        ap.h = hid_in;
        ap.gamma = static_cast<const __nv_bfloat16*>(h->w.W_attn_norm) + (size_t)layer * d;
        ap.a = h->Xp;
        ap.goff = h->goff_attn;
        ap.qkv = h->qkv;
        ap.err = h->dev_err;
        ap.out = h->attn_out;
        e = h->timed(K_ATTN, st, [&] { return launch_attn_norm(ap, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("attention norm: ") + cudaGetErrorString(e));
        GemmLaunch qg{};
        qg.tmA = &h->tmXp;
        qg.tmB = &h->tmWqkv[layer];
        qg.goff = h->goff_attn;
        qg.first_group = 0;
        qg.ngroups = 1;
        qg.K = d;
        qg.n_tiles_n = h->nqkv / 256;
        qg.b_rows_per_group = h->nqkv;
        qg.epi_mode = EPI_ROPE;
        qg.rope = h->rope;
        qg.rope_S = c.attn_seq;
        qg.rope_dh = c.head_dim;
        qg.n_rot = (c.attn_heads + c.attn_kv_heads) * c.head_dim;
        qg.out = h->qkv;
        qg.ldo = h->nqkv;
        qg.vt = h->vt;
        qg.vt_rows = c.attn_kv_heads * c.head_dim;
        qg.err = h->dev_err;
        qg.tmB_pair = pair_gemm(T) ? &h->tmWqkvp[layer] : nullptr;
        qg.sched = h->sched_for(layer, SCHED_QKV, d);
        e = h->timed(K_ATTN_GEMM, st, [&] { return launch_grouped_gemm(qg, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("qkv gemm: ") + cudaGetErrorString(e));
        // q/k/v rows of this call only: a sequence's 128-row box reads zeros past T
        // (never stale or uninitialised rows, which the masked products would
        // still multiply by zero).
        CUtensorMap tm_qkv, tm_vt;
        const uint64_t vt_rows = (uint64_t)((T + c.attn_seq - 1) / c.attn_seq) * c.attn_kv_heads * c.head_dim;
        if (!make_tmap(&tm_qkv, h->qkv, h->nqkv, T, 128) ||
            !make_tmap(&tm_vt, h->vt, kVtSlots, vt_rows, (uint32_t)c.head_dim))
            return h->fail(TRIMMOE_ERR_CUDA, "attention: cuTensorMapEncodeTiled failed");
        e = h->timed(K_ATTN, st, [&] { return launch_attention(ap, &tm_qkv, &tm_vt, c.head_dim, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("attention: ") + cudaGetErrorString(e));
        GemmLaunch og = qg;
        og.rope = nullptr;
        og.tmA = &h->tmAttn;
        og.tmB = &h->tmWo[layer];
        og.tmB_pair = pair_gemm(T) ? &h->tmWop[layer] : nullptr;
        og.K = hd;
        og.n_tiles_n = d / 256;
        og.b_rows_per_group = d;
        og.epi_mode = EPI_RESID;
        og.out = h->hm;
        og.ldo = d;
        og.res = hid_in;
        og.ldr = d;
        og.sched = h->sched_for(layer, SCHED_O, hd);
        e = h->timed(K_ATTN_GEMM, st, [&] { return launch_grouped_gemm(og, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("output projection: ") + cudaGetErrorString(e));
        h->launches += 4;
        h->flops_attn_gemm += 2.0 * T * d * (double)h->nqkv + 2.0 * T * (double)hd * d;
        double pairs = 0.0;                      // causal (query, key) pairs
        for (int t0 = 0; t0 < T; t0 += c.attn_seq) {
            const double n = std::min(c.attn_seq, T - t0);
            pairs += n * (n + 1) / 2;
        }
        h->flops_attn += 4.0 * c.head_dim * (double)c.attn_heads * pairs;
        hid = h->hm;
        if (out && out->h_attn) {
            e = cudaMemcpyAsync(out->h_attn, h->hm, (size_t)T * d * 2, cudaMemcpyDeviceToDevice, st);
            if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "copy h_attn failed");
        }
    }

    RouterParams rp;
    rp.T = T;
    rp.d = d;
    rp.n_out = n_out;
    rp.n_lo = E;
    rp.ng = router_pass_rows(n_out);
    rp.nl = router_lo_rows(E, rp.ng);
    rp.zs = n_out;
    rp.ksplit = router_ksplit(T, d, n_out, h->num_sms);
    rp.h = hid;
    rp.alive = tok->alive;
    rp.Bhi = h->rt_hi + (size_t)layer * n_out * d;
    rp.Blo = h->rt_lo + (size_t)layer * E * d;
    rp.zpart = h->zbuf;
    rp.sqpart = h->sqbuf;
    rp.err = h->dev_err;
    // With the attention sublayer the router rows read h_mid while the exit-head
    // and centroid rows read the state entering the layer: two passes.
    RouterParams rx = rp;
    if (has_attn) {
        rp.n_out = E;
        rp.ng = router_pass_rows(E);
        rp.nl = router_lo_rows(E, rp.ng);
        rx.h = hid_in;
        rx.n_out = n_out - E;
        rx.n_lo = 0;
        rx.ng = router_pass_rows(n_out - E);
        rx.nl = 0;
        rx.Bhi = rp.Bhi + (size_t)E * d;
        rx.zpart = h->zbuf + E;
        rx.sqpart = h->sqbuf_x;
    }
    dp.zpart = h->zbuf;
    dp.sqpart = h->sqbuf;
    dp.sqpart_x = has_attn ? h->sqbuf_x : nullptr;
    dp.bias = h->rt_bias + (size_t)layer * n_out;
    dp.zs = n_out;
    dp.ksplit = rp.ksplit;
    dp.use_norm = gamma != nullptr;
    dp.norm_eps = c.norm_eps;
    dp.rnorm = h->rnorm;
    dp.has_head = layer > 0;
    dp.n_cent = Kc;
    dp.cnorm = h->cnorm + (size_t)layer * Kc;
    dp.lhat_tab = h->lhat + (size_t)layer * Kc;
    dp.lhat_out = (out && out->lhat) ? out->lhat : nullptr;
    const int top_full = std::min(c.H - 1, c.N - 1 - layer);
    const int n_thr = h->thr_off[layer + 1] - h->thr_off[layer];
    const int n_depth = h->tab_depths[layer];
    // Tables built for every layer at the start of the forward serve any T;
    // a layer that builds its own pays off once the tokens outnumber them.
    const bool shared_tabs = n_depth > 0 && (h->tabs_ready || (size_t)(n_thr + 1) * n_depth * 4 <= (size_t)T);
    const size_t tab_off = h->la_all ? (size_t)h->h_la[layer].tab_off : 0;
    dp.phi_tabs = shared_tabs ? h->phi_tabs + tab_off : nullptr;
    dp.dbar_shared = h->dbar_shared;
    dp.thr = h->thr + h->thr_off[layer];
    dp.n_thr = n_thr;
    dp.dmin = top_full - n_depth + 1;
    dp.phi_tabs_out = h->phi_tabs + tab_off;
    dp.dbar_shared_out = h->dbar_shared;
    dp.la_scratch = shared_tabs ? h->la_scratch : nullptr;
    dp.calib = h->calib;
    dp.prev_target = h->prev_target;
    dp.c_trans = h->c_counts;
    dp.c_alive = dp.c_trans + (size_t)std::max(c.N - 1, 1) * E * E;
    dp.c_resid = dp.c_alive + c.N;
    dp.c_act = dp.c_resid + (size_t)c.N * c.M;
    dp.c_above = dp.c_act + (size_t)c.N * E;
    dp.s = tok->s;
    dp.Dhat = tok->Dhat;
    dp.Dbar = tok->Dbar;
    dp.pJ = tok->pJ;
    dp.alive = tok->alive;
    dp.last_exec = tok->last_exec;
    dp.xi_last = tok->xi_last;
    dp.exit_layer = tok->exit_layer;
    dp.topk_idx = (out && out->topk_idx) ? out->topk_idx : h->topk_idx;
    dp.topk_g = (out && out->topk_g) ? out->topk_g : h->topk_g;
    dp.I_out = (out && out->I) ? out->I : h->I;
    dp.xi_out = (out && out->xi) ? out->xi : h->xi;
    dp.action = (out && out->action) ? out->action : h->action;
    dp.exp_sel = (out && out->exp_sel) ? out->exp_sel : h->exp_sel;
    dp.srv_sel = (out && out->srv_sel) ? out->srv_sel : h->srv_sel;
    dp.tab.cand_m = h->cand_m;
    dp.tab.cand_k = h->cand_k;
    dp.tab.cand_Q = h->cand_Q;
    dp.tab.cand_off = h->cand_off;
    dp.tab.ctab = h->ctab;
    dp.tab.max_layer_cand = h->max_layer_cand;
    dp.tab.trans = h->trans;
    dp.tab.comp = h->comp;
    dp.tab.P = h->P;
    dp.tab.theta = h->theta;
    dp.tab.lambda = h->lambda;
    dp.tab.eps = h->eps;
    dp.ctr = h->ctr;

    // Shared look-ahead tables: light ones (M*E <= 256) on the side stream,
    // overlapping the router; heavy ones in line after it (run beside the
    // issue-bound router they slowed it more than they saved: Qwen-shaped,
    // M*E = 600, 23.5 -> 24.7 ms per forward; Switch-shaped 1.47 -> 1.40 ms).
    // Already built for every layer at the start of the forward?
    const bool tabs_here = shared_tabs && !h->tabs_ready;
    const bool tabs_aside = tabs_here && c.M * E <= 256;
    if (tabs_aside) {
        e = cudaEventRecord(h->ev_fork, st);
        if (e == cudaSuccess) e = cudaStreamWaitEvent(h->aux, h->ev_fork, 0);
        if (e == cudaSuccess) e = launch_lookahead_shared(dp, n_depth, h->aux);
        if (e == cudaSuccess) e = cudaEventRecord(h->ev_join, h->aux);
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("look-ahead tables: ") + cudaGetErrorString(e));
    }
    // Hidden rows for the router's TMA loads (128-token x 64-column boxes).
    CUtensorMap tm_h, tm_hx;
    if (T > 0 && (!make_tmap(&tm_h, rp.h, d, T, 128) || (has_attn && !make_tmap(&tm_hx, rx.h, d, T, 128))))
        return h->fail(TRIMMOE_ERR_CUDA, "router: cuTensorMapEncodeTiled failed");
    e = h->timed(K_ROUTER, st, [&] {
        cudaError_t e2 = launch_router(&tm_h, &h->tmRhi[layer], &h->tmRlo[layer], rp, h->num_sms, st);
        return (e2 == cudaSuccess && has_attn)
                   ? launch_router(&tm_hx, &h->tmRxhi[layer], nullptr, rx, h->num_sms, st)
                   : e2;
    });
    if (has_attn) h->launches += 1;
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("router: ") + cudaGetErrorString(e));
    if (tabs_aside) {
        e = cudaStreamWaitEvent(st, h->ev_join, 0);
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("look-ahead join: ") + cudaGetErrorString(e));
    }
    e = h->timed(K_DECIDE, st, [&] {
        cudaError_t e2 = (tabs_here && !tabs_aside) ? launch_lookahead_shared(dp, n_depth, st) : cudaSuccess;
        return e2 == cudaSuccess ? launch_decide(dp, h->num_sms, st) : e2;
    });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("decide: ") + cudaGetErrorString(e));

    CompactParams cp;
    cp.T = T;
    cp.k = K;
    cp.E = E;
    cp.has_shared = has_sh;
    cp.nblk = (T + 255) / 256;
    cp.action = dp.action;
    cp.exp_sel = dp.exp_sel;
    cp.blk_counts = h->blk_counts;
    cp.goff = h->goff;
    cp.perm = h->perm;
    cp.pos_pair = h->pos_pair;
    cp.pos_sh = h->pos_sh;
    cp.ctr = h->ctr;
    e = h->timed(K_COMPACT, st, [&] { return launch_compact(cp, st); });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("compact: ") + cudaGetErrorString(e));
    const int max_rows = T * K + (has_sh ? T : 0);
    e = h->timed(K_GATHER, st, [&] {
        return launch_gather(h->perm, h->goff, E, K, d, hid, h->rnorm, gamma, h->Xp, max_rows, h->num_sms, st);
    });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("gather: ") + cudaGetErrorString(e));

    GemmLaunch g1{};
    g1.tmA = &h->tmXp;
    g1.tmB = &h->tmW13[layer];
    // Routed experts: with at least kTransposedMinRows rows per expert the
    // down projection (and the up projection of ReLU experts) runs on the
    // transposed pair kernel, tokens on the MMA's N side so that a group's
    // last tile pads at most 15 tokens; SwiGLU up projections run on the pair
    // kernel for large groups and the single-CTA kernel otherwise;
    // decode-sized batches split K on the single-CTA kernel.
    const bool pair_routed = pair_gemm((long long)T * K / E);
    const bool relu = c.act != 1;
    const bool transposed = (long long)T * K / E >= kTransposedMinRows;
    g1.transposed = relu && transposed;
    g1.tmB_pair = (g1.transposed || pair_routed) ? &h->tmW13p[layer] : nullptr;
    g1.goff = h->goff;
    g1.first_group = 0;
    g1.ngroups = E;
    g1.a_rebase = 0;
    g1.out_rebase = 0;
    g1.K = d;
    g1.n_tiles_n = (int)(F13 / 256);
    g1.b_rows_per_group = (int)F13;
    g1.epi_mode = c.act == 1 ? EPI_SWIGLU : EPI_RELU;
    g1.out = h->act;
    g1.ldo = c.F;
    g1.err = h->dev_err;
    g1.sched = h->sched_for(layer, SCHED_UP, d);
    // Few executed pairs (decode-sized batches): few tiles would leave most
    // CTAs idle, so the K range is split and a finish kernel adds the parts.
    const bool small = (long long)T * K <= kSplitKRows;
    const int est_groups = (int)std::min<long long>(E, (long long)T * K);
    if (small) {
        g1.ksplit = grouped_gemm_ksplit(est_groups * g1.n_tiles_n, d / 64, h->num_sms);
        g1.partial = h->splitk;
        g1.ldp = g1.n_tiles_n * 256;
        g1.pstride = (size_t)kSplitKRows * g1.ldp;
    }
    e = h->timed(K_GEMM_UP, st, [&] {
        cudaError_t e2 = launch_grouped_gemm(g1, h->num_sms, st);
        return (e2 == cudaSuccess && g1.ksplit > 1) ? launch_splitk_finish(g1, h->num_sms, st) : e2;
    });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("gemm up: ") + cudaGetErrorString(e));
    GemmLaunch g2 = g1;
    g2.tmA = &h->tmAct;
    g2.tmB = &h->tmW2[layer];
    g2.transposed = transposed;
    g2.sched = h->sched_for(layer, SCHED_DOWN, c.F);
    g2.tmB_pair = (g2.transposed || pair_routed) ? &h->tmW2p[layer] : nullptr;
    g2.K = c.F;
    g2.n_tiles_n = d / 256;
    g2.b_rows_per_group = d;
    g2.epi_mode = EPI_STORE;
    g2.out = h->Y;
    g2.ldo = d;
    g2.ksplit = small ? grouped_gemm_ksplit(est_groups * g2.n_tiles_n, c.F / 64, h->num_sms) : 1;
    g2.ldp = g2.n_tiles_n * 256;
    g2.pstride = (size_t)kSplitKRows * g2.ldp;
    e = h->timed(K_GEMM_DOWN, st, [&] {
        cudaError_t e2 = launch_grouped_gemm(g2, h->num_sms, st);
        return (e2 == cudaSuccess && g2.ksplit > 1) ? launch_splitk_finish(g2, h->num_sms, st) : e2;
    });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("gemm down: ") + cudaGetErrorString(e));
    h->n_gemm_up++;
    h->n_gemm_down++;
    // router, decide, count (more than 256 tokens), scatter, gather, gate/up GEMM, down GEMM
    // (+ look-ahead tables, split-K finishes)
    h->launches += (T > 256 ? 7 : 6) + (tabs_here ? 1 : 0) + (g1.ksplit > 1 ? 1 : 0) + (g2.ksplit > 1 ? 1 : 0);
    if (has_sh) {
        GemmLaunch s1 = g1;
        s1.ksplit = 1;
        s1.transposed = 0;
        s1.tmB = &h->tmW13sh[layer];
        s1.tmB_pair = pair_gemm(T) ? &h->tmW13shp[layer] : nullptr;
        s1.first_group = E;
        s1.ngroups = 1;
        s1.out_rebase = 1;
        s1.n_tiles_n = 2 * c.F_sh / 256;
        s1.b_rows_per_group = 2 * c.F_sh;
        s1.epi_mode = EPI_SWIGLU;
        s1.out = h->act_sh;
        s1.ldo = c.F_sh;
        s1.sched = h->sched_for(layer, SCHED_SH_UP, d);
        e = h->timed(K_GEMM_UP, st, [&] { return launch_grouped_gemm(s1, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("shared gemm up: ") + cudaGetErrorString(e));
        GemmLaunch s2 = s1;
        s2.tmA = &h->tmActSh;
        s2.tmB = &h->tmW2sh[layer];
        s2.tmB_pair = pair_gemm(T) ? &h->tmW2shp[layer] : nullptr;
        s2.a_rebase = 1;
        s2.K = c.F_sh;
        s2.n_tiles_n = d / 256;
        s2.b_rows_per_group = d;
        s2.epi_mode = EPI_STORE;
        s2.out = h->Ysh;
        s2.ldo = d;
        s2.sched = h->sched_for(layer, SCHED_SH_DOWN, c.F_sh);
        e = h->timed(K_GEMM_DOWN, st, [&] { return launch_grouped_gemm(s2, h->num_sms, st); });
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("shared gemm down: ") + cudaGetErrorString(e));
        h->n_gemm_up++;
        h->n_gemm_down++;
        h->launches += 2;
    }

    CombineParams bp;
    bp.T = T;
    bp.d = d;
    bp.k = K;
    bp.renorm = c.renorm_topk;
    bp.has_shared = has_sh;
    bp.h = static_cast<__nv_bfloat16*>(tok->hidden);  // combine writes h in place
    bp.h_src = hid;                                    // residual base: h, or h_mid of the full block
    bp.action = dp.action;
    bp.topk_g = dp.topk_g;
    bp.pos_pair = h->pos_pair;
    bp.pos_sh = h->pos_sh;
    bp.Y = h->Y;
    bp.Ysh = h->Ysh;
    e = h->timed(K_COMBINE, st, [&] { return launch_combine(bp, h->num_sms, st); });
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("combine: ") + cudaGetErrorString(e));
    h->launches += 1;

    if (out && out->perm) {
        e = cudaMemcpyAsync(out->perm, h->perm, ((size_t)T * K + T) * 4, cudaMemcpyDeviceToDevice, st);
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "copy perm failed");
    }
    if (out && out->group_off) {
        e = cudaMemcpyAsync(out->group_off, h->goff, (size_t)(E + 2) * 4, cudaMemcpyDeviceToDevice, st);
        if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "copy group_off failed");
    }
    h->layer_calls++;
    h->win_ref_slots += (double)T * K;
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_layer_step(trimmoe_handle h, int layer, int T, trimmoe_tokens* tok,
                                             trimmoe_layer_out* out, void* stream) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (layer < 0 || layer >= h->cfg.N) return h->fail(TRIMMOE_ERR_ARG, "layer_step: layer out of range");
    if (T < 0 || T > h->cfg.T_max) return h->fail(TRIMMOE_ERR_ARG, "layer_step: T outside [0, T_max]");
    trimmoe_status s = check_tokens(h, tok);
    if (s != TRIMMOE_OK) return s;
    DeviceGuard g(h->dev);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    h->last_stream = st;
    if (T == 0) return TRIMMOE_OK;
    if (h->sched_any &&
        cudaMemsetAsync(h->gemm_sched + (size_t)layer * SCHED_SLOTS, 0, SCHED_SLOTS * sizeof(int), st) != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, "layer_step: tile counter reset failed");
    return layer_step_impl(h, layer, T, tok, out, st);
}

// Every layer's shared look-ahead tables in one launch (they depend only on
// the tables, the budget Dbar[0] and the cost weights, none of which change
// within a forward).  One launch per forward costs less than the tokens'
// own tables at any T (at one token: a table chain per layer on the critical
// path).  False if no layer has tables.
static bool build_all_tables(trimmoe_handle h, int T, const trimmoe_tokens* tok, cudaStream_t st, cudaError_t* err) {
    *err = cudaSuccess;
    if (!h->la_all || T <= 0) return false;
    bool any = false;
    for (const LaLayer& L : h->h_la) any |= L.n_depth > 0;
    if (!any) return false;
    const trimmoe_config& c = h->cfg;
    DecideParams dp{};
    dp.T = T;
    dp.N = c.N;
    dp.E = c.E;
    dp.M = c.M;
    dp.H = c.H;
    dp.omega_T = c.omega_T;
    dp.omega_D = c.omega_D;
    dp.Dbar = tok->Dbar;
    dp.thr = h->thr;
    dp.phi_tabs_out = h->phi_tabs;
    dp.dbar_shared_out = h->dbar_shared;
    dp.tab.cand_m = h->cand_m;
    dp.tab.cand_k = h->cand_k;
    dp.tab.cand_Q = h->cand_Q;
    dp.tab.cand_off = h->cand_off;
    dp.tab.ctab = h->ctab;
    dp.tab.max_layer_cand = h->max_layer_cand;
    dp.tab.P = h->P;
    dp.tab.eps = h->eps;
    *err = h->timed(K_DECIDE, st, [&] {
        return launch_lookahead_all(dp, h->la_layers, c.N, h->la_max_thr, h->la_max_depth, st);
    });
    if (*err != cudaSuccess) return false;
    h->launches += 1;
    return true;
}

static trimmoe_status forward_layers(trimmoe_handle h, int T, trimmoe_tokens* tok, cudaStream_t st) {
    // Tile counters of the layers' transposed pair GEMM launches start at zero.
    cudaError_t e = cudaSuccess;
    if (h->sched_any) e = cudaMemsetAsync(h->gemm_sched, 0, (size_t)SCHED_SLOTS * h->cfg.N * sizeof(int), st);
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("forward: ") + cudaGetErrorString(e));
    h->tabs_ready = build_all_tables(h, T, tok, st, &e);
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("look-ahead tables: ") + cudaGetErrorString(e));
    trimmoe_status s = TRIMMOE_OK;
    for (int l = 0; l < h->cfg.N && s == TRIMMOE_OK; ++l) s = layer_step_impl(h, l, T, tok, nullptr, st);
    h->tabs_ready = false;
    return s;
}

static bool same_tokens(const trimmoe_tokens& a, const trimmoe_tokens& b) {
    return a.hidden == b.hidden && a.s == b.s && a.Dhat == b.Dhat && a.Dbar == b.Dbar && a.pJ == b.pJ &&
           a.alive == b.alive && a.last_exec == b.last_exec && a.xi_last == b.xi_last && a.exit_layer == b.exit_layer;
}

// Captures the whole forward into gi (nothing runs); the host counters it
// would add are kept per replay.
static trimmoe_status capture_forward(trimmoe_handle h, int T, trimmoe_tokens* tok, cudaStream_t st, GraphInst& gi) {
    const uint64_t l0 = h->launches, c0 = h->layer_calls, u0 = h->n_gemm_up, d0 = h->n_gemm_down;
    const double fa0 = h->flops_attn, fg0 = h->flops_attn_gemm;
    h->cap_evs = &gi.evs;
    cudaGraph_t graph = nullptr;
    cudaError_t e = cudaStreamBeginCapture(st, cudaStreamCaptureModeThreadLocal);
    trimmoe_status s = TRIMMOE_OK;
    if (e == cudaSuccess) {
        s = forward_layers(h, T, tok, st);
        e = cudaStreamEndCapture(st, &graph);
    }
    h->cap_evs = nullptr;
    ForwardGraph& fg = h->fg;
    fg.launches = h->launches - l0;
    fg.layer_calls = h->layer_calls - c0;
    fg.n_gemm_up = h->n_gemm_up - u0;
    fg.n_gemm_down = h->n_gemm_down - d0;
    fg.flops_attn = h->flops_attn - fa0;
    fg.flops_attn_gemm = h->flops_attn_gemm - fg0;
    h->launches = l0;
    h->layer_calls = c0;
    h->n_gemm_up = u0;
    h->n_gemm_down = d0;
    h->flops_attn = fa0;
    h->flops_attn_gemm = fg0;
    if (e == cudaSuccess && s == TRIMMOE_OK) e = cudaGraphInstantiate(&gi.exec, graph, 0);
    if (graph) cudaGraphDestroy(graph);
    if (s != TRIMMOE_OK) return s;
    if (e != cudaSuccess) {
        cudaGetLastError();
        return h->fail(TRIMMOE_ERR_CUDA, std::string("forward: graph capture failed: ") + cudaGetErrorString(e));
    }
    return TRIMMOE_OK;
}

static trimmoe_status run_forward(trimmoe_handle h, int T, trimmoe_tokens* tok, cudaStream_t st) {
    NvtxRange range("trimmoe.forward");
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    const bool capturable = h->cfg.graphs && st != nullptr && st != cudaStreamLegacy && st != cudaStreamPerThread &&
                            cudaStreamIsCapturing(st, &cs) == cudaSuccess && cs == cudaStreamCaptureStatusNone;
    if (!capturable) return forward_layers(h, T, tok, st);
    ForwardGraph& fg = h->fg;
    if (fg.T != T || fg.st != st || !same_tokens(fg.tok, *tok)) {
        h->drop_graph();
        fg.T = T;
        fg.st = st;
        fg.tok = *tok;
    }
    if (fg.eager_runs < 1) {            // the first forward of a key runs eagerly (lazy set-up happens there)
        fg.eager_runs++;
        return forward_layers(h, T, tok, st);
    }
    if (!fg.inst[0].exec) {
        for (GraphInst& gi : fg.inst) {
            trimmoe_status s = capture_forward(h, T, tok, st, gi);
            if (s != TRIMMOE_OK) {
                h->drop_graph();
                return s;
            }
        }
    }
    GraphInst& gi = fg.inst[fg.next];
    h->read_graph_inst(gi);
    if (cudaGraphLaunch(gi.exec, st) != cudaSuccess) {
        cudaGetLastError();
        return h->fail(TRIMMOE_ERR_CUDA, "forward: graph launch failed");
    }
    gi.pending = h->cfg.profile != 0;
    fg.next ^= 1;
    h->launches += fg.launches;
    h->layer_calls += fg.layer_calls;
    h->n_gemm_up += fg.n_gemm_up;
    h->n_gemm_down += fg.n_gemm_down;
    h->flops_attn += fg.flops_attn;
    h->flops_attn_gemm += fg.flops_attn_gemm;
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_forward(trimmoe_handle h, int T, trimmoe_tokens* tok, void* stream) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (T < 0 || T > h->cfg.T_max) return h->fail(TRIMMOE_ERR_ARG, "forward: T outside [0, T_max]");
    trimmoe_status s = check_tokens(h, tok);
    if (s != TRIMMOE_OK) return s;
    DeviceGuard g(h->dev);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    h->last_stream = st;
    if (T == 0) return TRIMMOE_OK;
    return run_forward(h, T, tok, st);
}

extern "C" trimmoe_status trimmoe_forward_host(trimmoe_handle h, int T, trimmoe_tokens* tok, void* stream) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (T < 0 || T > h->cfg.T_max) return h->fail(TRIMMOE_ERR_ARG, "forward_host: T outside [0, T_max]");
    if (!tok || !tok->hidden || !tok->s || !tok->Dhat || !tok->Dbar || !tok->pJ || !tok->alive ||
        !tok->last_exec || !tok->xi_last || !tok->exit_layer)
        return h->fail(TRIMMOE_ERR_ARG, "forward_host: NULL pointer");
    DeviceGuard g(h->dev);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    h->last_stream = st;
    const size_t Tm = h->cfg.T_max;
    trimmoe_tokens& dt = h->dtok;
    if (!dt.hidden) {
        __nv_bfloat16* hid = nullptr;
        bool ok = h->dalloc(&hid, Tm * h->cfg.d) && h->dalloc(&dt.s, Tm) && h->dalloc(&dt.Dhat, Tm) &&
                  h->dalloc(&dt.Dbar, Tm) && h->dalloc(&dt.pJ, Tm) && h->dalloc(&dt.alive, Tm) &&
                  h->dalloc(&dt.last_exec, Tm) && h->dalloc(&dt.xi_last, Tm) && h->dalloc(&dt.exit_layer, Tm);
        dt.hidden = hid;
        if (!ok) {
            dt.hidden = nullptr;
            return h->fail(TRIMMOE_ERR_OOM, "forward_host: device allocation failed");
        }
    }
    const size_t n = (size_t)T;
    struct Cp { void* dst; const void* src; size_t bytes; };
    const Cp in[] = {{dt.hidden, tok->hidden, n * h->cfg.d * 2}, {dt.s, tok->s, n}, {dt.Dhat, tok->Dhat, n * 4},
                     {dt.Dbar, tok->Dbar, n * 4}, {dt.pJ, tok->pJ, n * 4}, {dt.alive, tok->alive, n},
                     {dt.last_exec, tok->last_exec, n}, {dt.xi_last, tok->xi_last, n * 4},
                     {dt.exit_layer, tok->exit_layer, n * 2}};
    for (const Cp& c : in)
        if (cudaMemcpyAsync(c.dst, c.src, c.bytes, cudaMemcpyHostToDevice, st) != cudaSuccess)
            return h->fail(TRIMMOE_ERR_CUDA, "forward_host: host-to-device copy failed");
    if (T > 0) {
        trimmoe_status s = run_forward(h, T, &dt, st);
        if (s != TRIMMOE_OK) return s;
    }
    for (const Cp& c : in)
        if (cudaMemcpyAsync(const_cast<void*>(c.src), c.dst, c.bytes, cudaMemcpyDeviceToHost, st) != cudaSuccess)
            return h->fail(TRIMMOE_ERR_CUDA, "forward_host: device-to-host copy failed");
    if (cudaStreamSynchronize(st) != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "forward_host: sync failed");
    int derr = 0;
    cudaMemcpy(&derr, h->dev_err, sizeof(int), cudaMemcpyDeviceToHost);
    if (derr) return h->fail(TRIMMOE_ERR_DEVICE_TIMEOUT, "forward_host: a kernel timed out waiting");
    return TRIMMOE_OK;
}

// Sum of the device counter copies (copy order; the ratio is a maximum).
cudaError_t read_counters(const DevCounters* dev, DevCounters* out) {
    DevCounters c[kCtrCopies];
    const cudaError_t e = cudaMemcpy(c, dev, sizeof c, cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return e;
    std::memset(out, 0, sizeof *out);
    for (int i = 0; i < kCtrCopies; ++i) {
        out->layer_tokens += c[i].layer_tokens;
        out->exec_tokens += c[i].exec_tokens;
        out->skipped += c[i].skipped;
        out->exited += c[i].exited;
        out->pairs_local_exact += c[i].pairs_local_exact;
        out->pairs_local_sub += c[i].pairs_local_sub;
        out->pairs_remote_exact += c[i].pairs_remote_exact;
        out->pairs_remote_sub += c[i].pairs_remote_sub;
        out->shared_rows += c[i].shared_rows;
        out->remote_hops += c[i].remote_hops;
        out->pairs_total += c[i].pairs_total;
        out->experts_touched += c[i].experts_touched;
        out->shared_touched += c[i].shared_touched;
        out->lookahead_shared += c[i].lookahead_shared;
        out->delay_ms += c[i].delay_ms;
        out->max_budget_ratio_bits = std::max(out->max_budget_ratio_bits, c[i].max_budget_ratio_bits);
    }
    return cudaSuccess;
}

extern "C" trimmoe_status trimmoe_stats(trimmoe_handle h, trimmoe_stats_t* out) {
    if (!h || !out) return TRIMMOE_ERR_ARG;
    DeviceGuard g(h->dev);
    if (cudaStreamSynchronize(h->last_stream) != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, std::string("stats: ") + cudaGetErrorString(cudaGetLastError()));
    DevCounters dc;
    int derr = 0;
    if (read_counters(h->ctr, &dc) != cudaSuccess ||
        cudaMemcpy(&derr, h->dev_err, sizeof derr, cudaMemcpyDeviceToHost) != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, "stats: copy failed");
    h->drain_events();
    const trimmoe_config& c = h->cfg;
    std::memset(out, 0, sizeof *out);
    out->layer_tokens = dc.layer_tokens;
    out->exec_tokens = dc.exec_tokens;
    out->skipped = dc.skipped;
    out->exited = dc.exited;
    out->pairs_local_exact = dc.pairs_local_exact;
    out->pairs_local_sub = dc.pairs_local_sub;
    out->pairs_remote_exact = dc.pairs_remote_exact;
    out->pairs_remote_sub = dc.pairs_remote_sub;
    out->shared_rows = dc.shared_rows;
    out->delay_ms = dc.delay_ms;
    out->remote_hops = (double)dc.remote_hops;
    float r;
    std::memcpy(&r, &dc.max_budget_ratio_bits, 4);
    out->max_budget_ratio = r;
    out->device_error = derr;
    out->launches = h->launches;
    out->layer_calls = h->layer_calls;
    const double n13F = (double)h->n13 * c.F;
    out->flops_gemm_up = 2.0 * dc.pairs_total * n13F * c.d + 2.0 * dc.shared_rows * 2.0 * c.F_sh * c.d;
    out->flops_gemm_down = 2.0 * dc.pairs_total * (double)c.d * c.F + 2.0 * dc.shared_rows * (double)c.d * c.F_sh;
    out->gemm_flops = out->flops_gemm_up + out->flops_gemm_down;
    const double dd = c.d, FF = c.F, Fs = c.F_sh;
    out->bytes_gemm_up = 2.0 * ((double)dc.experts_touched * n13F * dd + (double)dc.shared_touched * 2.0 * Fs * dd +
                                (double)dc.pairs_total * (dd + FF) + (double)dc.shared_rows * (dd + Fs));
    out->bytes_gemm_down = 2.0 * ((double)dc.experts_touched * dd * FF + (double)dc.shared_touched * dd * Fs +
                                  (double)dc.pairs_total * (FF + dd) + (double)dc.shared_rows * (Fs + dd));
    out->ms_decide = h->ms[K_DECIDE];
    out->ms_compact = h->ms[K_COMPACT];
    out->ms_gather = h->ms[K_GATHER];
    out->ms_gemm_up = h->ms[K_GEMM_UP];
    out->ms_gemm_down = h->ms[K_GEMM_DOWN];
    out->ms_combine = h->ms[K_COMBINE];
    out->ms_router = h->ms[K_ROUTER];
    out->lookahead_shared = dc.lookahead_shared;
    out->ms_attn = h->ms[K_ATTN];
    out->ms_attn_gemm = h->ms[K_ATTN_GEMM];
    out->flops_attn = h->flops_attn;
    out->flops_attn_gemm = h->flops_attn_gemm;
    out->n_gemm_up = h->n_gemm_up;
    out->n_gemm_down = h->n_gemm_down;
    out->pairs_executed = dc.pairs_total;
    out->bytes_expert_weights = 2.0 * ((double)dc.experts_touched * (n13F + FF) * dd +
                                       (double)dc.shared_touched * 3.0 * Fs * dd);
    if (derr) return h->fail(TRIMMOE_ERR_DEVICE_TIMEOUT, "stats: a kernel timed out waiting");
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_reset_stats(trimmoe_handle h) {
    if (!h) return TRIMMOE_ERR_ARG;
    DeviceGuard g(h->dev);
    if (cudaStreamSynchronize(h->last_stream) != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "reset: sync failed");
    h->drain_events();
    if (cudaMemset(h->ctr, 0, sizeof(DevCounters) * kCtrCopies) != cudaSuccess ||
        cudaMemset(h->dev_err, 0, sizeof(int)) != cudaSuccess ||
        cudaMemset(h->gemm_sched, 0, (size_t)SCHED_SLOTS * h->cfg.N * sizeof(int)) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, "reset: memset failed");
    for (double& m : h->ms) m = 0.0;
    h->launches = h->layer_calls = h->n_gemm_up = h->n_gemm_down = 0;
    h->flops_attn = h->flops_attn_gemm = 0.0;
    h->win_delay0 = 0.0;
    h->win_ref_slots = 0.0;
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_watchdog_selftest(trimmoe_handle h, int timeout_us, void* stream) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (timeout_us < 1 || timeout_us > 1000000) return h->fail(TRIMMOE_ERR_ARG, "watchdog_selftest: timeout_us out of range");
    DeviceGuard g(h->dev);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    h->last_stream = st;
    if (launch_watchdog_selftest(h->dev_err, (uint64_t)timeout_us * 1000ull, st) != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, std::string("watchdog_selftest: ") + cudaGetErrorString(cudaGetLastError()));
    h->launches += 1;
    int derr = 0;
    if (cudaStreamSynchronize(st) != cudaSuccess ||
        cudaMemcpy(&derr, h->dev_err, sizeof derr, cudaMemcpyDeviceToHost) != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, std::string("watchdog_selftest: ") + cudaGetErrorString(cudaGetLastError()));
    if (derr) return h->fail(TRIMMOE_ERR_DEVICE_TIMEOUT, "watchdog_selftest: a device wait ran out (code " +
                                                              std::to_string(derr) + ")");
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_calibration_begin(trimmoe_handle h) {
    if (!h) return TRIMMOE_ERR_ARG;
    DeviceGuard g(h->dev);
    if (cudaStreamSynchronize(h->last_stream) != cudaSuccess ||
        cudaMemset(h->c_counts, 0, h->n_counts * sizeof(unsigned long long)) != cudaSuccess ||
        cudaMemset(h->prev_target, 0xFF, (size_t)h->cfg.T_max * sizeof(int16_t)) != cudaSuccess ||
        cudaDeviceSynchronize() != cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, "calibration_begin: reset failed");
    h->drop_graph();      // the decision kernel's parameters change
    h->calib = 1;
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_calibration_end(trimmoe_handle h, long long T_cal, trimmoe_calibration_t* out) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (!out || T_cal < 0) return h->fail(TRIMMOE_ERR_ARG, "calibration_end: NULL output or negative T_cal");
    DeviceGuard g(h->dev);
    std::vector<unsigned long long> cnt(h->n_counts);
    if (cudaStreamSynchronize(h->last_stream) != cudaSuccess ||
        cudaMemcpy(cnt.data(), h->c_counts, cnt.size() * sizeof(unsigned long long), cudaMemcpyDeviceToHost) !=
            cudaSuccess)
        return h->fail(TRIMMOE_ERR_CUDA, "calibration_end: copy failed");
    h->drop_graph();
    h->calib = 0;
    const int N = h->cfg.N, E = h->cfg.E, M = h->cfg.M, K = h->cfg.k;
    const size_t ntr = (size_t)std::max(N - 1, 1) * E * E;
    const unsigned long long* trans = cnt.data();
    const unsigned long long* alive = trans + ntr;
    const unsigned long long* resid = alive + N;
    const unsigned long long* act = resid + (size_t)N * M;
    const unsigned long long* above = act + (size_t)N * E;
    auto put = [](uint64_t* dst, const unsigned long long* src, size_t n) {
        if (dst) for (size_t i = 0; i < n; ++i) dst[i] = src[i];
    };
    put(out->trans, trans, ntr);
    put(out->alive, alive, N);
    put(out->resid, resid, (size_t)N * M);
    put(out->act, act, (size_t)N * E);
    put(out->above, above, (size_t)N * E);
    if (out->P)
        for (int l = 0; l + 1 < N; ++l)
            for (int k = 0; k < E; ++k) {
                unsigned long long tot = 0;
                for (int kp = 0; kp < E; ++kp) tot += trans[((size_t)l * E + k) * E + kp];
                for (int kp = 0; kp < E; ++kp)
                    out->P[((size_t)l * E + k) * E + kp] =
                        tot ? (float)((double)trans[((size_t)l * E + k) * E + kp] / (double)tot) : (float)(1.0 / E);
            }
    for (int l = 0; l < N; ++l) {
        const double a = (double)alive[l];
        const float pi = T_cal > 0 ? (float)(a / (double)T_cal) : 0.0f;
        if (out->pi) out->pi[l] = pi;
        for (int k = 0; k < E; ++k) {
            const double routed = (double)act[(size_t)l * E + k];
            const float sg = routed > 0 ? (float)((double)above[(size_t)l * E + k] / routed) : 0.0f;
            const float af = a > 0 ? (float)(routed / (K * a)) : 0.0f;
            if (out->sigma) out->sigma[(size_t)l * E + k] = sg;
            if (out->act_freq) out->act_freq[(size_t)l * E + k] = af;
            if (out->lambda) out->lambda[(size_t)l * E + k] = pi * sg * af;
        }
        if (out->rho)
            for (int m = 0; m < M; ++m)
                out->rho[(size_t)l * M + m] = a > 0 ? (float)((double)resid[(size_t)l * M + m] / a) : 0.0f;
    }
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_replicate(int N, int E, int M, const float* lambda, const float* rho,
                                            const float* trans, const double* expert_bytes, const double* capacity,
                                            uint16_t* place, int* added) {
    if (N < 1 || E < 1 || M < 1 || M > 16 || !lambda || !rho || !trans || !expert_bytes || !capacity || !place) {
        tmoe::set_global_error("replicate: bad dimensions or NULL pointer");
        return TRIMMOE_ERR_ARG;
    }
    const uint32_t mmask = (M >= 16) ? 0xFFFFu : ((1u << M) - 1u);
    std::vector<double> used(M, 0.0);
    for (int l = 0; l < N; ++l)
        for (int k = 0; k < E; ++k) {
            if ((place[(size_t)l * E + k] & mmask) == 0) {
                tmoe::set_global_error("replicate: an expert has no server (Eq. 2)");
                return TRIMMOE_ERR_COVERAGE;
            }
            for (int m = 0; m < M; ++m)
                if ((place[(size_t)l * E + k] >> m) & 1u) used[m] += expert_bytes[(size_t)l * E + k];
        }
    int n_added = 0;
    while (true) {
        double best = -1.0;
        int bm = -1, bl = -1, bk = -1;
        for (int m = 0; m < M; ++m)
            for (int l = 0; l < N; ++l)
                for (int k = 0; k < E; ++k) {
                    const uint16_t mask = place[(size_t)l * E + k];
                    if ((mask >> m) & 1u) continue;
                    if (used[m] + expert_bytes[(size_t)l * E + k] > capacity[m]) continue;
                    double sum = 0.0;
                    int hosts = 0;
                    for (int mp = 0; mp < M; ++mp)
                        if ((mask >> mp) & 1u) { sum += (double)trans[(size_t)m * M + mp]; ++hosts; }
                    const double reach = hosts ? sum / hosts : 0.0;
                    const double b = (double)lambda[(size_t)l * E + k] * (double)rho[(size_t)l * M + m] * reach;
                    if (b > best) { best = b; bm = m; bl = l; bk = k; }
                }
        if (bm < 0) break;
        place[(size_t)bl * E + bk] |= (uint16_t)(1u << bm);
        used[bm] += expert_bytes[(size_t)bl * E + bk];
        ++n_added;
    }
    if (added) *added = n_added;
    return TRIMMOE_OK;
}

extern "C" trimmoe_status trimmoe_feedback(trimmoe_handle h, const trimmoe_feedback_cfg* fb, int T,
                                           trimmoe_tokens* tok, trimmoe_feedback_out* out, void* stream) {
    if (!h) return TRIMMOE_ERR_ARG;
    if (!fb || !out) return h->fail(TRIMMOE_ERR_ARG, "feedback: NULL argument");
    if (fb->user_size < 1 || !(fb->eta >= 0.f) || !std::isfinite(fb->eta) || !(fb->p_min >= 0.f) ||
        !(fb->p_min <= 1.f) || !(fb->kappa >= 0.f) || !std::isfinite(fb->kappa))
        return h->fail(TRIMMOE_ERR_ARG, "feedback: need user_size >= 1, eta >= 0, 0 <= p_min <= 1, kappa >= 0");
    if (T < 0 || T > h->cfg.T_max) return h->fail(TRIMMOE_ERR_ARG, "feedback: T outside [0, T_max]");
    trimmoe_status s = check_tokens(h, tok);
    if (s != TRIMMOE_OK) return s;
    DeviceGuard g(h->dev);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    h->last_stream = st;
    FeedbackParams p;
    p.T = T;
    p.N = h->cfg.N;
    p.user_size = fb->user_size;
    p.users = (T + fb->user_size - 1) / fb->user_size;
    p.eta = fb->eta;
    p.p_min = fb->p_min;
    p.pJ = tok->pJ;
    p.alive = tok->alive;
    p.exit_layer = tok->exit_layer;
    p.xi_last = tok->xi_last;
    p.Dhat = tok->Dhat;
    p.Dbar = tok->Dbar;
    p.util = h->fb_util;
    p.updated = h->fb_updated;
    p.result = h->fb_result;
    cudaError_t e = launch_feedback(p, st);
    if (e == cudaSuccess) e = cudaStreamSynchronize(st);
    double res[2] = {0.0, 0.0};
    DevCounters dc;
    if (e == cudaSuccess) e = cudaMemcpy(res, h->fb_result, sizeof res, cudaMemcpyDeviceToHost);
    if (e == cudaSuccess) e = read_counters(h->ctr, &dc);
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, std::string("feedback: ") + cudaGetErrorString(e));
    const double window_delay = dc.delay_ms - h->win_delay0;
    const double ref = h->win_ref_slots;
    const double D_util = res[0];
    const double T_norm = (ref > 0.0) ? window_delay / (ref * (double)h->cfg.d_ref_ms) : 0.0;
    double wD = (double)h->cfg.omega_D + (double)fb->kappa * (D_util - T_norm);
    wD = std::min(std::max(wD, 0.0), 1.0);
    trimmoe_config c2 = h->cfg;
    c2.omega_D = (float)wD;
    c2.omega_T = 1.0f - c2.omega_D;
    const std::vector<float> ctab = delay_cost_table(c2, h->h_trans, h->h_comp);
    e = cudaMemcpy(h->ctab, ctab.data(), ctab.size() * sizeof(float), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return h->fail(TRIMMOE_ERR_CUDA, "feedback: table upload failed");
    h->cfg = c2;
    h->win_delay0 = dc.delay_ms;
    h->win_ref_slots = 0.0;
    h->drop_graph();      // omega enters the decision kernel by value
    out->omega_T = c2.omega_T;
    out->omega_D = c2.omega_D;
    out->T_norm = T_norm;
    out->D_util = D_util;
    out->users_updated = (int)res[1];
    out->window_delay_ms = window_delay;
    out->window_ref_slots = ref;
    return TRIMMOE_OK;
}

extern "C" const char* trimmoe_last_error(trimmoe_handle h) {
    if (!h) {
        std::lock_guard<std::mutex> g(g_err_mu);
        return g_create_error.c_str();
    }
    return h->err.c_str();
}

extern "C" void trimmoe_destroy(trimmoe_handle h) {
    if (!h) return;
    DeviceGuard g(h->dev);
    cudaDeviceSynchronize();
    h->drain_events();
    h->drop_graph();
    for (cudaEvent_t e : h->ev_free) cudaEventDestroy(e);
    if (h->ev_fork) cudaEventDestroy(h->ev_fork);
    if (h->ev_join) cudaEventDestroy(h->ev_join);
    if (h->aux) cudaStreamDestroy(h->aux);
    for (void* p : h->allocs) cudaFree(p);
    delete h;
}
