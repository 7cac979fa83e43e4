/*
 * trimmoe.h -- C ABI of the GB300 (sm_103a) adaptive-depth MoE layer step.
 *
 * The library implements the per-token, per-layer online decision of the
 * paper's Sec. V (Algorithm 2 / Table II) together with the MoE computation it
 * gates: router and importance (Eq. 4), exit-head confidence (Eq. 7-9), skip
 * test (Eq. 5, 34, 35), substitute-or-fetch with server choice and look-ahead
 * (Eq. 30-31, 38-40), state updates (Eq. 41-42), compaction of the executed
 * (token, expert) pairs, grouped expert FFN and the gate-weighted combine.
 * The M edge servers of Sec. III-A are simulated by the placement and cost
 * tables only.
 *
 * Conventions for every call:
 *  - Functions never abort or throw; they return a trimmoe_status and
 *    trimmoe_last_error() gives a one-line reason for the handle's last error.
 *  - "device" pointers are CUDA device memory owned by the caller; they must
 *    stay valid until the work queued on the stream has finished.  "host"
 *    tables are copied during trimmoe_create and may be freed afterwards.
 *  - bf16 values are IEEE bfloat16 bit patterns (uint16).  All arrays are
 *    dense, row-major, with the shapes given in brackets.
 *  - Layers, experts, servers and tokens are 0-based.
 *  - Calls are asynchronous on the given stream (a cudaStream_t passed as
 *    void*, NULL = legacy default stream) except trimmoe_stats,
 *    trimmoe_forward_host and trimmoe_watchdog_selftest, which synchronise.  A handle must not be used by
 *    two streams or two host threads at the same time: its workspaces are
 *    shared by all its calls.
 */
#ifndef TRIMMOE_H
#define TRIMMOE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    TRIMMOE_OK = 0,
    TRIMMOE_ERR_ARG = -1,            /* null / misaligned pointer, bad size or layer */
    TRIMMOE_ERR_UNSUPPORTED = -2,    /* dimensions this build does not handle */
    TRIMMOE_ERR_OOM = -3,            /* device allocation failed */
    TRIMMOE_ERR_CUDA = -4,           /* a CUDA runtime/driver call failed */
    TRIMMOE_ERR_COVERAGE = -5,       /* an expert has no server (violates Eq. 2) */
    TRIMMOE_ERR_DEVICE_TIMEOUT = -6  /* a kernel gave up waiting and flagged it */
} trimmoe_status;

typedef struct trimmoe* trimmoe_handle;

/* Actions written to trimmoe_layer_out.action (Sec. V-A). */
/* Which bounded device wait ran out first (trimmoe_stats_t.device_error).
 * Every wait of a kernel on an mbarrier or a flag has a time limit; the first
 * one to run out writes its code, makes the other roles of its CTA return, and
 * the kernel ends normally, so the CUDA context stays usable. */
enum {
    TRIMMOE_DEVERR_NONE = 0,
    TRIMMOE_DEVERR_GEMM_PRODUCER = 1,  /* grouped GEMM: TMA producer waiting for a free stage */
    TRIMMOE_DEVERR_GEMM_MMA = 2,       /* grouped GEMM: MMA issuer waiting for operands or TMEM */
    TRIMMOE_DEVERR_GEMM_EPILOGUE = 3,  /* grouped GEMM: epilogue waiting for an accumulator */
    TRIMMOE_DEVERR_ROUTER = 4,         /* router logits kernel */
    TRIMMOE_DEVERR_ATTENTION = 5,      /* attention kernel (including its softmax pair barriers) */
    TRIMMOE_DEVERR_SELFTEST = 6        /* trimmoe_watchdog_selftest */
};

enum { TRIMMOE_EXEC = 0, TRIMMOE_SKIP = 1, TRIMMOE_EXIT = 2, TRIMMOE_DEAD = 3 };

/* Model and policy hyper-parameters.
 *  N layers; d = d_model; E routed experts; k = top-k; F = routed expert d_ff;
 *  F_sh = shared-expert d_ff (0 = none; always SwiGLU, always local, Sec. III-B);
 *  C exit-head classes (1 = sigmoid head of Sec. IV-A, >1 = max softmax prob);
 *  M servers (<= 16); H look-ahead horizon (Eq. 39, 1 = myopic);
 *  act: 0 ReLU, 1 SwiGLU; renorm_topk: combine weights renormalised over the
 *  top-k (the importance I of Eq. 4 always uses the raw softmax gates);
 *  n_sub: substitutes per target (|R_{l,r}| <= n_sub, Sec. III-A);
 *  T_max: largest token count of a call (sizes the workspaces);
 *  omega_T, omega_D: weights of Eq. (21)/(31); d_ref_ms: d^ref of Eq. (31);
 *  phi_beta: Q = phi_beta * (1 - Sim)/2 (Eq. 3 with a linear phi);
 *  profile: 1 = record CUDA events around each kernel launch (trimmoe_stats
 *  then reports per-kernel device time); 2 = around the grouped GEMM launches
 *  only (each event pair inside a replayed graph costs a few microseconds);
 *  norm_eps: epsilon of the pre-FFN RMSNorm (used when W_norm != NULL);
 *  n_centroids: K_c centroids per layer for the token-similarity exit-point
 *  prediction of Eq. (36) (0 = off, at most 256);
 *  attn_heads, attn_kv_heads, head_dim, attn_seq, rope_theta: the attention
 *  sublayer of the full transformer block (attn_heads = 0: the MoE step
 *  alone).  With it every layer first runs, for every live token, pre-norm
 *  grouped-query causal attention: attn_heads query heads and attn_kv_heads
 *  key/value heads of head_dim, rotary embedding with base rope_theta, within
 *  sequences of attn_seq consecutive tokens (token t sits at position
 *  t mod attn_seq).  Attention stays local to the token's server (Sec. III-C,
 *  attention placement): a skip bypasses only the MoE sublayer;
 *  graphs: 1 = trimmoe_forward / trimmoe_forward_host replay the whole
 *  forward as a CUDA graph.  The first forward with a given (T, token
 *  buffers, stream) runs as plain launches; the next one captures the layer
 *  loop (twice, so profiling events of one replay can be read while the
 *  other runs) and every later one launches the graph.  Results are those of
 *  the plain launches.  Not used on the legacy or per-thread default stream,
 *  or when the stream is already being captured (the launches then go into
 *  the caller's capture); feedback and calibration calls drop the graph.
 * Supported: d % 256 == 0, d <= 16384; SwiGLU F % 128 == 0, ReLU F % 256 == 0;
 * F_sh % 128 == 0; E <= 128; k <= min(E, 8); C <= 256; M*E <= 1024; H <= 6;
 * n_sub <= 3; attention: head_dim 64 or 128, attn_heads % attn_kv_heads == 0,
 * (attn_heads + 2 attn_kv_heads) * head_dim % 256 == 0, 1 <= attn_seq <= 128,
 * W_norm required. */
typedef struct {
    int N, d, E, k, F, F_sh, C, M, H;
    int act;
    int renorm_topk;
    int n_sub;
    int T_max;
    float omega_T, omega_D, d_ref_ms, phi_beta;
    int profile;
    float norm_eps;
    int n_centroids;
    int attn_heads, attn_kv_heads, head_dim, attn_seq;
    float rope_theta;
    int graphs;
} trimmoe_config;

/* Weights (device, bf16 except the biases, borrowed; 16-byte aligned).
 *  W_r  [N][E][d], b_r fp32 [N][E]        router (Sec. III-B)
 *  W_x  [N][C][d], b_x fp32 [N][C]        exit heads h_l (Eq. 7)
 *  W13  [N][E][n13*F][d]   n13 = 2 (SwiGLU) or 1 (ReLU).  SwiGLU rows are
 *       interleaved in blocks of 128: rows [256b, 256b+128) are gate rows
 *       128b..128b+127 and rows [256b+128, 256b+256) the matching up rows.
 *  W2   [N][E][d][F]
 *  W13_sh [N][2*F_sh][d] (same interleave), W2_sh [N][d][F_sh]; NULL if F_sh == 0.
 *  W_norm [N][d] weights gamma_l of the MoE sublayer's pre-FFN RMSNorm, or NULL
 *       for none.  With it, layer l computes r = 1/sqrt(mean(h^2) + norm_eps);
 *       the router reads h*r*gamma_l (fp32), the experts its bf16 rounding, the
 *       exit head h*r, and the combine adds to h itself (pre-norm residual).
 *  centroids [N][K_c][d] (n_centroids > 0): representations entering layer l
 *       of the token-similarity reference set (Eq. 36); read at create.
 *  W_attn_norm [N][d], W_qkv [N][(Hq + 2 Hkv) Dh][d], W_o [N][d][Hq Dh]
 *       (attn_heads > 0): RMSNorm weights of the attention sublayer, the fused
 *       query/key/value projection (query heads, then key heads, then value
 *       heads, Dh rows each) and the output projection.  Layer l then computes
 *       a = bf16(h r' gamma'); v = bf16(a W_v^T); q and k are rotated (rotary
 *       embedding) in fp32 on the unrounded projection a W_q^T, a W_k^T and
 *       rounded to bf16 once, after the rotation; causal softmax attention (query head j reads key/value head
 *       j / (Hq/Hkv)), h_mid = bf16(h + o W_o^T); the router, experts and
 *       residual read h_mid, the exit head of layer l-1 and the exit prediction
 *       read h (the state entering the layer), and a token that exits at layer
 *       l keeps h. */
typedef struct {
    const void* W_r;
    const float* b_r;
    const void* W_x;
    const float* b_x;
    const void* W13;
    const void* W2;
    const void* W13_sh;
    const void* W2_sh;
    const void* W_norm;
    const void* centroids;
    const void* W_attn_norm;
    const void* W_qkv;
    const void* W_o;
} trimmoe_weights;

/* The paper's input tables (host, copied at create).
 *  place [N][E]    bit m set iff expert k of layer l is deployed on server m,
 *                  x_{m,l,k} of Eq. (1)-(2); every entry must be non-zero.
 *  sim   [N][E][E] Sim_l(r, k) of Eq. (3); R_{l,r} = the n_sub experts k != r of
 *                  highest Sim_l(r, k) with Sim >= sub_thresh[l] (ties: lower k).
 *  sub_thresh [N]
 *  trans_ms [M][M] z_l/B + tau between servers (Eq. 14); the diagonal is unused.
 *  comp_ms  [N][M] c_l / F_m (Eq. 15).
 *  P     [N-1][E][E] P_l(k -> k') (Eq. 38); rows sum to 1.  May be NULL if N == 1.
 *  theta [N] importance thresholds (Eq. 24); lambda [N] Lambda = lambda_l * I
 *  (Eq. 5); eps [N] per-layer skip tolerance (Eq. 25), used by the look-ahead. */
typedef struct {
    const uint16_t* place;
    const float* sim;
    const float* sub_thresh;
    const float* trans_ms;
    const float* comp_ms;
    const float* P;
    const float* theta;
    const float* lambda;
    const float* eps;
    const float* centroid_exit;
} trimmoe_tables;

/* Per-token state (device, borrowed, length >= T; updated in place).
 *  hidden bf16 [T][d] hidden states h, read and written in place;
 *  s current server (Eq. 29); Dhat accumulated degradation (Eq. 41-42);
 *  Dbar per-token budget (Eq. 33); pJ confidence requirement (Eq. 8);
 *  alive y (Eq. 6); last_exec 1 iff the previous layer executed (Eq. 9);
 *  xi_last last exit confidence evaluated; exit_layer first layer that did not
 *  run (N when the token ran every layer). */
typedef struct {
    void* hidden;
    uint8_t* s;
    float* Dhat;
    float* Dbar;
    float* pJ;
    uint8_t* alive;
    uint8_t* last_exec;
    float* xi_last;
    int16_t* exit_layer;
} trimmoe_tokens;

/* Optional per-layer outputs of trimmoe_layer_step (device; any may be NULL).
 *  topk_idx int32 [T][k] (-1 for dead tokens); topk_g fp32 [T][k] softmax gates;
 *  I fp32 [T]; xi fp32 [T] (-1 where not evaluated); action uint8 [T];
 *  exp_sel, srv_sel uint8 [T][k] executed expert and server (255 unless EXEC);
 *  perm int32 [T*k + T]: the executed pairs t*k+j ordered by (expert, t, j),
 *  then the tokens that run the shared expert (executed or skipped) by t;
 *  group_off int32 [E+2]: pairs of expert e are perm[group_off[e] ..
 *  group_off[e+1]), shared rows perm[group_off[E] .. group_off[E+1]);
 *  lhat int16 [T]: predicted exit layer (Eq. 36; N without prediction, -1 for
 *  dead tokens);
 *  h_attn bf16 [T][d] (full block only): the state after the attention
 *  sublayer, h_mid (rows of tokens that are not live are unspecified). */
typedef struct {
    int32_t* topk_idx;
    float* topk_g;
    float* I;
    float* xi;
    uint8_t* action;
    uint8_t* exp_sel;
    uint8_t* srv_sel;
    int32_t* perm;
    int32_t* group_off;
    int16_t* lhat;
    void* h_attn;
} trimmoe_layer_out;

/* Counters accumulated since create / the last reset (Fig. 5(b) categories). */
typedef struct {
    uint64_t layer_tokens;        /* live (token, layer) decisions */
    uint64_t exec_tokens;         /* token-layers executed */
    uint64_t skipped;             /* token-layers skipped */
    uint64_t exited;              /* exits */
    uint64_t pairs_local_exact;   /* executed (token, slot) pairs by kind */
    uint64_t pairs_local_sub;
    uint64_t pairs_remote_exact;
    uint64_t pairs_remote_sub;
    uint64_t shared_rows;         /* rows through the shared expert */
    double delay_ms;              /* sum of d(m, k) of Eq. (30) over executed pairs */
    double remote_hops;           /* executed pairs on a server other than s */
    float max_budget_ratio;       /* max Dhat / Dbar seen after a decision */
    int device_error;             /* 0, or the TRIMMOE_DEVERR_* code of the first wait that ran out */
    uint64_t launches;            /* kernels launched by the library */
    uint64_t layer_calls;         /* layers processed */
    double gemm_flops;            /* 2*M*N*K of the grouped FFN GEMMs that ran */
    /* Device time per kernel family in ms (profile != 0 only). */
    double ms_decide, ms_compact, ms_gather, ms_gemm_up, ms_gemm_down, ms_combine;
    uint64_t n_gemm_up, n_gemm_down;
    double flops_gemm_up, flops_gemm_down;
    double ms_router;             /* router / exit-head logits kernel (profile != 0) */
    /* Algorithmic HBM bytes of the grouped FFN GEMMs that ran: weights of the
     * experts that received work once, activation rows in and out. */
    double bytes_gemm_up, bytes_gemm_down;
    /* Decisions whose look-ahead table (Eq. 39) was read from the per-layer
     * tables shared by all tokens of equal budget instead of computed per token
     * (the results are the same either way). */
    uint64_t lookahead_shared;
    /* Attention sublayer of the full block: device time (profile != 0) of the
     * RMSNorm + attention kernels and of the two projection GEMMs, and their
     * FLOPs (projections 2*T*d*(Hq+2Hkv)Dh + 2*T*Hq*Dh*d; attention
     * 4*Dh*Hq*(causal query-key pairs)). */
    double ms_attn, ms_attn_gemm;
    double flops_attn, flops_attn_gemm;
    /* Executed (token, slot) pairs, and the bytes of the expert weights that
     * received work (each such expert's up and down projections once per
     * layer call, plus the shared expert's when it ran). */
    uint64_t pairs_executed;
    double bytes_expert_weights;
} trimmoe_stats_t;

/* Validate, copy the tables, derive the candidate lists V_{l,r} and losses Q,
 * allocate the workspaces for T_max tokens, and build the TMA descriptors.
 * Errors: ARG (null or misaligned pointer, non-stochastic P), UNSUPPORTED
 * (dimensions), COVERAGE (Eq. 2), OOM, CUDA.  *out is NULL on error. */
trimmoe_status trimmoe_create(const trimmoe_config* cfg, const trimmoe_weights* w,
                              const trimmoe_tables* tab, trimmoe_handle* out);

/* One MoE layer over tokens [0, T) (the per-layer body of Algorithm 2, plus the gated FFN and
 * combine).  Dead tokens are untouched.  0 <= layer < N, 0 <= T <= T_max.
 * out may be NULL.  Asynchronous on stream. */
trimmoe_status trimmoe_layer_step(trimmoe_handle h, int layer, int T, trimmoe_tokens* tok,
                                  trimmoe_layer_out* out, void* stream);

/* Layers 0..N-1 in order (the layer loop of Algorithm 2).  Asynchronous on stream. */
trimmoe_status trimmoe_forward(trimmoe_handle h, int T, trimmoe_tokens* tok, void* stream);

/* trimmoe_forward on HOST buffers: copies hidden and the token state to device
 * buffers owned by the handle, runs the forward, copies them back and
 * synchronises the stream.  Pointers in tok are host pointers (pinned memory
 * gives the fastest copies). */
trimmoe_status trimmoe_forward_host(trimmoe_handle h, int T, trimmoe_tokens* tok, void* stream);

/* Synchronise the handle's last stream and read the counters.  Returns
 * DEVICE_TIMEOUT if a kernel flagged one (the flag stays set until reset). */
trimmoe_status trimmoe_stats(trimmoe_handle h, trimmoe_stats_t* out);

/* Zero the counters and the device error flag (synchronises). */
trimmoe_status trimmoe_reset_stats(trimmoe_handle h);

/* Failure-detection self-check of the bounded device waits.  Launches one
 * kernel on stream whose mbarrier never receives an arrival: warp 0 waits on
 * it with a limit of timeout_us microseconds (1 ... 1000000), runs out, raises
 * the CTA's abort flag and writes TRIMMOE_DEVERR_SELFTEST to the handle's
 * device error word; warp 1 waits on the same barrier with the kernels' normal
 * two-second limit and returns as soon as it sees the abort.  The call then
 * synchronises the stream and reads the word back.
 * Returns DEVICE_TIMEOUT when the wait ran out as designed (the flag stays set,
 * and trimmoe_stats reports it, until trimmoe_reset_stats), OK if the word was
 * not set, ARG for a NULL handle or a limit out of range, CUDA if the launch
 * failed.  The handle stays usable afterwards. */
trimmoe_status trimmoe_watchdog_selftest(trimmoe_handle h, int timeout_us, void* stream);

/* Last error message of the handle ("" if none); NULL handle: the last error of
 * a call made without a handle (trimmoe_create, trimmoe_compact_noalloc). */
const char* trimmoe_last_error(trimmoe_handle h);

/* Free the handle and its workspaces (synchronises first).  NULL is a no-op. */
void trimmoe_destroy(trimmoe_handle h);

/* Runtime feedback between forwards (the periodic update of Algorithm 2): the exit-threshold
 * update of Eq. (37) and the dual-weight update of Eq. (43).
 *  user_size: users are blocks of user_size consecutive tokens (Eq. 33);
 *  eta, p_min: step and floor of Eq. (37); kappa: step of Eq. (43). */
typedef struct {
    int user_size;
    float eta, p_min, kappa;
} trimmoe_feedback_cfg;

typedef struct {
    float omega_T, omega_D;       /* weights after the update (used by later calls) */
    double T_norm;                /* observed normalised delay of the window */
    double D_util;                /* observed budget utilisation of the window */
    int users_updated;            /* users whose p_J moved (had exits in the window) */
    double window_delay_ms;       /* summed per-step delay d(m,k) of the window's executions */
    double window_ref_slots;      /* token x layer x slot count of the window's calls */
} trimmoe_feedback_out;

/* End an observation window.  For each user with exits in the window (tokens
 * with alive == 0 and exit_layer < N; xi_last is the confidence that admitted
 * the exit), every token's pJ (device, in place) becomes
 * clamp(pJ + eta * (mean exit confidence - pJ), p_min, 1)  (Eq. 37).
 * D_util = mean over users of sum(Dhat)/sum(Dbar); T_norm = window delay /
 * (window_ref_slots * d_ref), the window's delay over the full-depth exact
 * reference; omega_D = clamp(omega_D + kappa * (D_util - T_norm), 0, 1),
 * omega_T = 1 - omega_D (Eq. 43); the handle uses the new weights from the
 * next call on.  The window is everything since the previous trimmoe_feedback
 * or trimmoe_reset_stats; call it after a forward and before the token state is
 * re-initialised.  Synchronises the stream.  ERR_ARG on a bad configuration. */
trimmoe_status trimmoe_feedback(trimmoe_handle h, const trimmoe_feedback_cfg* fb, int T, trimmoe_tokens* tok,
                                trimmoe_feedback_out* out, void* stream);

/* Offline stage (Algorithm 1) on calibration runs.
 * Between trimmoe_calibration_begin and trimmoe_calibration_end every layer step
 * counts, per live token: activity (pi_l, Eq. 26), its server before the layer
 * (rho_{m,l}), each routed slot (activation frequency a_l^k), each slot with
 * I > theta_l (sigma_l^k, Eq. 27), and the transition of its slot-0 target from
 * the previous layer (Eq. 38; a token's first layer only records its target).
 * Results (host arrays owned by the caller, any may be NULL):
 *  counts: trans [N-1][E][E], alive [N], resid [N][M], act [N][E], above [N][E];
 *  P [N-1][E][E] = row-normalised transitions (uniform rows without data);
 *  pi [N] = alive / T_cal; sigma [N][E] = above / act (0 without data);
 *  act_freq [N][E] = act / (k * alive); lambda [N][E] = pi * sigma * act_freq;
 *  rho [N][M] = resid / alive. */
typedef struct {
    uint64_t *trans, *alive, *resid, *act, *above;
    float *P, *pi, *sigma, *act_freq, *lambda, *rho;
} trimmoe_calibration_t;

/* Zero the counts and start counting (synchronises). */
trimmoe_status trimmoe_calibration_begin(trimmoe_handle h);

/* Stop counting and write the counts and statistics; T_cal = number of
 * calibration tokens that entered layer 0 (synchronises). */
trimmoe_status trimmoe_calibration_end(trimmoe_handle h, long long T_cal, trimmoe_calibration_t* out);

/* Greedy communication-aware replication (Algorithm 1, Eq. 28), host only.
 * place [N][E] server masks (updated in place; every entry non-zero); lambda,
 * rho as above; trans [M][M] delays; expert_bytes [N][E] memory of one copy;
 * capacity [M] bytes.  The benefit of a copy of expert k of layer l on a server
 * m without it is lambda_l^k * rho_{m,l} * mean over its current hosts m' of
 * trans[m][m']; each step places the feasible copy (fits the residual memory
 * of m, Eq. c.1) of largest benefit, ties to the lowest (m, l, k), until none is
 * feasible.  *added receives the number of copies placed.  ERR_ARG on bad input,
 * ERR_COVERAGE if an expert has no server on entry. */
trimmoe_status trimmoe_replicate(int N, int E, int M, const float* lambda, const float* rho, const float* trans,
                                 const double* expert_bytes, const double* capacity, uint16_t* place, int* added);

/* Compaction of one layer's decisions without any device allocation (the
 * paper has no counterpart: this entry point exists for callers that cannot
 * call cudaMalloc, e.g. code running inside an allocator callback or in a
 * process whose device memory is entirely owned by another pool).
 * Inputs (device): action uint8 [T] and exp_sel uint8 [T][k] as written by
 * trimmoe_layer_step.  Outputs (device, caller-owned): perm int32 [T*k + T] and
 * group_off int32 [E+2] with the same contents as trimmoe_layer_out, pos_pair
 * int32 [T*k] (position of pair t*k+j in perm, -1 if not executed) and pos_sh
 * int32 [T] (row of token t among the shared-expert rows, -1 if none; may be
 * NULL when has_shared == 0).  Per-chunk scratch lives in one static device
 * array of about 132 KB held by every GPU that loads the library until exit;
 * hence T <= 65536 and E <= 128 (ERR_ARG beyond, with a message in
 * trimmoe_last_error(NULL)).  It calls no cudaMalloc/cudaFree.  The first call on
 * each device looks up the array's device address once (cudaGetSymbolAddress)
 * and keeps it; make that first call before any stream capture.  After
 * cudaDeviceReset the device gets a new context in which the array may sit
 * elsewhere: the next call notices the new context and looks the address up
 * again, so the first call after a reset must also come before any capture.
 * All calls share the array and it keeps the previous call's contents (the
 * call clears what must start at zero): calls whose work overlaps on the GPU
 * (other streams, other host threads) race and must be serialised by the
 * caller.  Asynchronous on stream. */
trimmoe_status trimmoe_compact_noalloc(const uint8_t* action, const uint8_t* exp_sel, int T, int k, int E,
                                       int has_shared, int32_t* perm, int32_t* group_off,
                                       int32_t* pos_pair, int32_t* pos_sh, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* TRIMMOE_H */
