// TrimMoE online stage -- CPU oracle.
//
// TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
// restatement of the paper's online stage (Sec. V, Algorithm 2 / Table II) that
// the CUDA library is checked against.  Only the tests, the smoke check and the
// benchmark's CPU-baseline leg may load it.  It shares no code, header, table or
// constant with the CUDA path.
//
// Precision: dot products accumulate in double; every decision quantity (gates,
// importance, costs, look-ahead, budgets) is fp32 with one fixed operation order.
// Build with -ffp-contract=off so no multiply-add is fused.
//
// Readings of the paper where it is silent or garbled (each one is listed with
// its reason in the design notes):
//  * the MoE sublayer is pre-norm (as in the three evaluated models): with norm
//    weights gamma_l the router and the experts read x = h * r * gamma_l,
//    r = 1/sqrt(mean(h^2) + eps); the exit head reads h * r; the residual is h.
//    The router uses x unrounded, the experts its bf16 rounding;
//  * importance I = sum of the full-softmax probabilities of the top-k set (Eq. 4);
//  * a NaN logit ranks as -infinity;
//  * top-k is ordered by logit, descending, ties to the lower expert index;
//  * exit head: C == 1 -> sigmoid (Sec. IV-A); C > 1 -> max softmax probability;
//  * exit is an action at layer l, admissible iff l > 0, layer l-1 was executed
//    and xi_{l-1} >= p_J (Eq. 8, 9, 34); layers >= l then do not run;
//  * Q = phi((1 - Sim)/2) with phi(x) = beta * x; R_{l,r} = the n_sub most similar
//    k != r with Sim >= sub_thresh[l] (Eq. 3);
//  * skip loss Lambda = lambda_l * I (Eq. 5 with a linear rho);
//  * top-k > 1: slots are decided in slot order; one skip decision per layer;
//    Gamma = sum over slots of the per-slot minimum transmission (Eq. 35);
//    the token moves to slot 0's server; only slot 0 carries the look-ahead;
//  * look-ahead (Eq. 39): budget frozen at R = Dbar - Dhat; future location = the
//    server of the future action; future target k' ~ P_l(k_exec -> .); future skip
//    costs omega_D * eps_l' / Dbar and is admitted iff no budget-feasible candidate
//    is local and eps_l' <= R; exit is not modelled inside the look-ahead; zero
//    beyond the last layer;
//  * action choice (Eq. 40): ties go EXEC, then SKIP, then EXIT; exit only when the
//    best alternative's total is > 0 (Sec. V-A);
//  * full block (optional): the attention sublayer runs for every live token
//    before the MoE decision (Sec. III-C: a skip bypasses only the FFN); the
//    router reads its output, the exit head of layer l-1 the state entering
//    layer l; a token exiting at layer l leaves with that entering state.
#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <vector>
#ifdef _OPENMP
#include <omp.h>
#endif

namespace {

const float kInf = std::numeric_limits<float>::infinity();
const int kGateUpGroup = 128;   // W13 row interleave of the gate / up projections

enum { A_EXEC = 0, A_SKIP = 1, A_EXIT = 2, A_DEAD = 3 };

inline float bf2f(uint16_t b) {
    uint32_t u = (uint32_t)b << 16;
    float f;
    std::memcpy(&f, &u, 4);
    return f;
}

inline uint16_t f2bf(float f) {       // round to nearest even
    uint32_t u;
    std::memcpy(&u, &f, 4);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu)) return 0x7FC0;
    u += 0x7FFFu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

inline uint16_t d2bf(double v) { return f2bf((float)v); }

double dot_bf16(const uint16_t* a, const uint16_t* b, int n) {
    double acc = 0.0;
    for (int i = 0; i < n; ++i) acc += (double)bf2f(a[i]) * (double)bf2f(b[i]);
    return acc;
}

}  // namespace

extern "C" {

// Model hyper-parameters and the paper's input tables (all host memory).
typedef struct {
    int N, d, E, k, F, F_sh, C, M, H, act, renorm_topk, n_sub;
    float omega_T, omega_D, d_ref, phi_beta, norm_eps;
    const uint16_t* place;     // [N][E] server bit mask, x_{m,l,k} (Eq. 1-2)
    const float* sim;          // [N][E][E] Sim_l(r, k) (Eq. 3)
    const float* sub_thresh;   // [N] substitute admission threshold on Sim
    const float* trans;        // [M][M] z/B + tau in ms (Eq. 14)
    const float* comp;         // [N][M] c_l / F_m in ms (Eq. 15)
    const float* P;            // [N-1][E][E] P_l(k -> k') (Eq. 38)
    const float* theta;        // [N] importance thresholds (Eq. 24)
    const float* lambda_;      // [N] slope of Lambda = lambda * I (Eq. 5)
    const float* eps;          // [N] per-layer skip tolerance (Eq. 25)
    int n_centroids;           // K_c centroids per layer for Eq. (36); 0 = no exit prediction
    // Attention sublayer of the full block (attn_heads = 0: the MoE step alone).
    int attn_heads, attn_kv_heads, head_dim, attn_seq;
    float rope_theta;
} OrModel;

// Weights of one layer (host, bf16 bits).
typedef struct {
    const uint16_t* W_r;       // [E][d] router
    const float* b_r;          // [E]
    const uint16_t* W_x_prev;  // [C][d] exit head of layer l-1 (NULL at l = 0)
    const float* b_x_prev;     // [C]
    const uint16_t* W13;       // [E][n13*F][d], gate/up interleaved by 128 rows
    const uint16_t* W2;        // [E][d][F]
    const uint16_t* W13_sh;    // [2*F_sh][d] or NULL
    const uint16_t* W2_sh;     // [d][F_sh] or NULL
    const uint16_t* W_norm;    // [d] RMSNorm weights of this layer, NULL = no normalisation
    const uint16_t* centroids; // [K_c][d] representations entering this layer (Eq. 36)
    const float* centroid_exit;// [K_c] average exit layer of each centroid's calibration tokens
    const uint16_t* W_attn_norm; // [d] RMSNorm weights in front of the attention sublayer
    const uint16_t* W_qkv;     // [(Hq + 2 Hkv) Dh][d]: query heads, then key heads, then value heads
    const uint16_t* W_o;       // [d][Hq Dh]
} OrLayerWeights;

// Per-token state (host arrays of length T), updated in place.
typedef struct {
    uint8_t* s;          // current server s_{i,q,l} (Eq. 29)
    float* Dhat;         // accumulated degradation (Eq. 41-42)
    float* Dbar;         // per-token budget (Eq. 33)
    float* pJ;           // confidence requirement
    uint8_t* alive;      // y_{i,q,l} (Eq. 6)
    uint8_t* last_exec;  // 1 iff the previous layer was executed
    float* xi_last;      // last exit confidence computed
    int16_t* exit_layer; // first layer not run (N = full depth)
} OrTokens;

// Per-layer outputs (host); any pointer may be NULL.
typedef struct {
    int32_t* topk_idx;   // [T][k]
    float* topk_g;       // [T][k] full-softmax gates
    float* I;            // [T]
    float* xi;           // [T] (-1 when not evaluated)
    uint8_t* action;     // [T]
    uint8_t* exp_sel;    // [T][k]
    uint8_t* srv_sel;    // [T][k]
    int32_t* perm;       // [T*k + T] routed pairs (t*k+j) by expert, then shared rows (t)
    int32_t* group_off;  // [E+2]
    uint8_t* near;       // [T] near-threshold bits
    float* Gamma;        // [T]
    float* tot_exec;     // [T]
    float* tot_skip;     // [T] (+inf when skip not admitted)
    int16_t* lhat;       // [T] predicted exit layer (Eq. 36), N without prediction, -1 dead
} OrLayerOut;

// One token's decision at one layer.
typedef struct {
    int topk[16];
    float g[16];
    float I, xi, Gamma, tot_exec, tot_skip, Lambda;
    int action, skip_ok, exit_ok;
    int exp_sel[16], srv_sel[16];
    float Q_sel[16], f_sel[16];
    float Dhat_new;
    int s_new;
    int near;
    int Lhat;          // predicted exit layer (Eq. 36), or N without a prediction
} OrDecision;

// ---------------------------------------------------------------- routing

// RMS factor r = 1 / sqrt(mean(h^2) + eps) of the pre-FFN RMSNorm.
double or_rms_factor(const uint16_t* h, int d, float eps) {
    double ss = 0.0;
    for (int i = 0; i < d; ++i) ss += (double)bf2f(h[i]) * (double)bf2f(h[i]);
    return 1.0 / std::sqrt(ss / d + (double)eps);
}

// Router logits on the normalised hidden state, softmax and top-k; importance
// by Eq. (4).  W_norm == NULL: the router reads h itself.
void or_router(const OrModel* md, const uint16_t* W_r, const float* b_r, const uint16_t* W_norm,
               const uint16_t* h, float* z, float* p, int* topk, float* g, float* I) {
    const int E = md->E, d = md->d;
    if (W_norm) {
        const double r = or_rms_factor(h, d, md->norm_eps);
        for (int e = 0; e < E; ++e) {
            const uint16_t* w = W_r + (size_t)e * d;
            double acc = 0.0;
            for (int i = 0; i < d; ++i)
                acc += (double)bf2f(h[i]) * (double)bf2f(W_norm[i]) * (double)bf2f(w[i]);
            z[e] = (float)(acc * r) + b_r[e];
        }
    } else {
        for (int e = 0; e < E; ++e) z[e] = (float)dot_bf16(h, W_r + (size_t)e * d, d) + b_r[e];
    }
    for (int e = 0; e < E; ++e)
        if (z[e] != z[e]) z[e] = -kInf;
    float zmax = -kInf;
    for (int e = 0; e < E; ++e) zmax = std::max(zmax, z[e]);
    float S = 0.0f;
    for (int e = 0; e < E; ++e) { p[e] = expf(z[e] - zmax); S = S + p[e]; }
    for (int e = 0; e < E; ++e) p[e] = p[e] / S;
    std::vector<char> used(E, 0);
    for (int j = 0; j < md->k; ++j) {
        int best = -1;
        for (int e = 0; e < E; ++e)
            if (!used[e] && (best < 0 || z[e] > z[best])) best = e;   // ties: lower index
        used[best] = 1;
        topk[j] = best;
    }
    float acc = 0.0f;
    for (int j = 0; j < md->k; ++j) { g[j] = p[topk[j]]; acc = acc + g[j]; }
    *I = acc;
}

// Exit-head confidence xi = h_l(h) in [0, 1] (Eq. 7).  C == 1: sigmoid head of
// Sec. IV-A; C > 1: the largest softmax probability over C classes.  With
// normalise != 0 the head reads the RMS-normalised state h * r.
float or_exit_conf(const OrModel* md, const uint16_t* W_x, const float* b_x, const uint16_t* h,
                   int normalise, float* logits_out) {
    const int C = md->C, d = md->d;
    const double r = normalise ? or_rms_factor(h, d, md->norm_eps) : 1.0;
    std::vector<float> x(C);
    for (int c = 0; c < C; ++c) x[c] = (float)(dot_bf16(h, W_x + (size_t)c * d, d) * r) + b_x[c];
    if (logits_out) for (int c = 0; c < C; ++c) logits_out[c] = x[c];
    if (C == 1) return 1.0f / (1.0f + expf(-x[0]));
    float xm = -kInf;
    for (int c = 0; c < C; ++c) xm = std::max(xm, x[c]);
    float S = 0.0f;
    for (int c = 0; c < C; ++c) S = S + expf(x[c] - xm);
    return 1.0f / S;
}

// ------------------------------------------------------- candidates / costs

// Substitution loss Q_l(r, k) of Eq. (3) with phi(x) = beta * x.
float or_sub_loss(const OrModel* md, int l, int r, int k) {
    if (k == r) return 0.0f;
    float s = md->sim[((size_t)l * md->E + r) * md->E + k];
    return md->phi_beta * ((1.0f - s) / 2.0f);
}

// Feasible execution set V_{l,r} = {r} U R_{l,r} (Sec. III-A), listed as
// (server, expert) pairs deployed per x_{m,l,k} (Eq. 11): the exact expert
// first, then substitutes by expert index; servers ascending within an expert.
int or_candidates(const OrModel* md, int l, int r, int* cm, int* ck, float* cQ, int cap) {
    const int E = md->E, M = md->M;
    std::vector<int> subs;
    for (int k = 0; k < E; ++k)
        if (k != r && md->sim[((size_t)l * E + r) * E + k] >= md->sub_thresh[l]) subs.push_back(k);
    std::stable_sort(subs.begin(), subs.end(), [&](int a, int b) {
        return md->sim[((size_t)l * E + r) * E + a] > md->sim[((size_t)l * E + r) * E + b];
    });
    if ((int)subs.size() > md->n_sub) subs.resize(md->n_sub);
    std::sort(subs.begin(), subs.end());
    std::vector<int> experts;
    experts.push_back(r);
    for (int k : subs) experts.push_back(k);
    int n = 0;
    for (int k : experts)
        for (int m = 0; m < M; ++m)
            if ((md->place[(size_t)l * E + k] >> m) & 1u) {
                if (n < cap) { cm[n] = m; ck[n] = k; cQ[n] = or_sub_loss(md, l, r, k); }
                ++n;
            }
    return n;
}

// Per-step delay d(m, k) of Eq. (30) from server s.
static float step_delay(const OrModel* md, int l, int s, int m) {
    float tr = (m != s) ? md->trans[(size_t)s * md->M + m] : 0.0f;
    return tr + md->comp[(size_t)l * md->M + m];
}

// Execute cost f(m, k) of Eq. (31).
float or_exec_cost(const OrModel* md, int l, int s, int m, float Q, float Dbar) {
    float c = md->omega_T * (step_delay(md, l, s, m) / md->d_ref);
    if (Q > 0.0f) c = c + md->omega_D * (Q / Dbar);
    return c;
}

// --------------------------------------------------------------- look-ahead

struct CandList { std::vector<int> m, k; std::vector<float> Q; };

static CandList cand_list(const OrModel* md, int l, int r) {
    int cap = md->M * md->E;
    CandList c;
    c.m.resize(cap); c.k.resize(cap); c.Q.resize(cap);
    int n = or_candidates(md, l, r, c.m.data(), c.k.data(), c.Q.data(), cap);
    c.m.resize(n); c.k.resize(n); c.Q.resize(n);
    return c;
}

// V^{(h)}_{lp}(m, k'): best next-layer action from server m for target k' (the
// inner minimum of Eq. 39).  phi_next = Phi^{(h-1)}_{lp} or NULL when it is zero.
static void value_table(const OrModel* md, int lp, float R, float Dbar, const float* phi_next,
                        float* V) {
    const int M = md->M, E = md->E;
    for (int kp = 0; kp < E; ++kp) {
        CandList c = cand_list(md, lp, kp);
        for (int m = 0; m < M; ++m) {
            float best = kInf;
            bool local = false;
            for (size_t i = 0; i < c.m.size(); ++i) {
                if (!(c.Q[i] <= R)) continue;
                float v = or_exec_cost(md, lp, m, c.m[i], c.Q[i], Dbar);
                if (phi_next) v = v + phi_next[c.m[i] * E + c.k[i]];
                best = std::min(best, v);
                if (c.m[i] == m) local = true;
            }
            if (!local && md->eps[lp] <= R) {
                float v = md->omega_D * (md->eps[lp] / Dbar);
                if (phi_next) v = v + phi_next[m * E + kp];
                best = std::min(best, v);
            }
            V[m * E + kp] = best;
        }
    }
}

// Phi^{(h)}_l(m, k) = sum_{k'} P_l(k -> k') V^{(h)}_{l+1}(m, k')  (Eq. 39).
static float phi_entry(const OrModel* md, int l, int m, int k, const float* V) {
    const int E = md->E;
    float acc = 0.0f;
    for (int kp = 0; kp < E; ++kp) acc = acc + md->P[((size_t)l * E + k) * E + kp] * V[m * E + kp];
    return acc;
}

// Phi^{(H-1)}_l(m, k) for every (m, k), evaluated bottom-up from the deepest
// future layer (memoised form of Eq. 39).  Zero when H == 1 or l is the last
// layer.  cap limits the future layers to l+1 .. l+cap (a predicted exit).
void or_lookahead_table_capped(const OrModel* md, int l, float R, float Dbar, int cap, float* phi_out) {
    const int M = md->M, E = md->E;
    const int top = std::min(std::min(md->H - 1, md->N - 1 - l), cap);
    std::vector<float> V(M * E), phi_next(M * E), phi_cur(M * E);
    bool have_next = false;
    for (int j = top; j >= 1; --j) {
        const int lp = l + j;
        value_table(md, lp, R, Dbar, have_next ? phi_next.data() : nullptr, V.data());
        for (int m = 0; m < M; ++m)
            for (int k = 0; k < E; ++k) phi_cur[m * E + k] = phi_entry(md, lp - 1, m, k, V.data());
        phi_next.swap(phi_cur);
        have_next = true;
    }
    for (int i = 0; i < M * E; ++i) phi_out[i] = have_next ? phi_next[i] : 0.0f;
}

void or_lookahead_table(const OrModel* md, int l, float R, float Dbar, float* phi_out) {
    or_lookahead_table_capped(md, l, R, Dbar, 1 << 30, phi_out);
}

// Token-similarity exit-point prediction (Eq. 36): the nearest centroid by
// cosine similarity (ties to the lower index) gives L_hat = round(mean exit
// layer of its calibration tokens), rounding halves up.  *best_score and *gap
// receive the best score and its margin over the second best (scores are the
// cosine similarities times |h|, which does not change the order).
int or_predict_exit(const OrModel* md, const uint16_t* centroids, const float* centroid_exit,
                    const uint16_t* h, float* best_score, float* gap) {
    const int K = md->n_centroids, d = md->d;
    int best = -1;
    float bs = 0.0f, second = -kInf;
    for (int j = 0; j < K; ++j) {
        const uint16_t* c = centroids + (size_t)j * d;
        double nn = 0.0;
        for (int i = 0; i < d; ++i) nn += (double)bf2f(c[i]) * (double)bf2f(c[i]);
        const float cn = (float)std::sqrt(nn);
        const float sc = (cn > 0.0f) ? (float)dot_bf16(h, c, d) / cn : -kInf;
        if (best < 0 || sc > bs) { second = (best < 0) ? -kInf : bs; best = j; bs = sc; }
        else if (sc > second) second = sc;
    }
    if (gap) *gap = bs - second;
    if (best_score) *best_score = bs;
    return (int)std::floor((double)centroid_exit[best] + 0.5);
}

static float value_naive(const OrModel* md, int lp, int h, int m, int kp, float R, float Dbar);

// Direct tree recursion of Eq. (39) without memoisation (pin for the table form).
float or_phi_naive(const OrModel* md, int l, int h, int m, int k, float R, float Dbar) {
    if (h == 0 || l >= md->N - 1) return 0.0f;
    float acc = 0.0f;
    for (int kp = 0; kp < md->E; ++kp) {
        float V = value_naive(md, l + 1, h, m, kp, R, Dbar);
        acc = acc + md->P[((size_t)l * md->E + k) * md->E + kp] * V;
    }
    return acc;
}

static float value_naive(const OrModel* md, int lp, int h, int m, int kp, float R, float Dbar) {
    CandList c = cand_list(md, lp, kp);
    const bool deeper = (h - 1 > 0) && (lp < md->N - 1);
    float best = kInf;
    bool local = false;
    for (size_t i = 0; i < c.m.size(); ++i) {
        if (!(c.Q[i] <= R)) continue;
        float v = or_exec_cost(md, lp, m, c.m[i], c.Q[i], Dbar);
        if (deeper) v = v + or_phi_naive(md, lp, h - 1, c.m[i], c.k[i], R, Dbar);
        best = std::min(best, v);
        if (c.m[i] == m) local = true;
    }
    if (!local && md->eps[lp] <= R) {
        float v = md->omega_D * (md->eps[lp] / Dbar);
        if (deeper) v = v + or_phi_naive(md, lp, h - 1, m, kp, R, Dbar);
        best = std::min(best, v);
    }
    return best;
}

// ------------------------------------------------------------ the decision

// One token, one layer: the per-token body of Algorithm 2, given the routing (topk, g, I) and
// the exit confidence xi (negative when not evaluated).
void or_decide_given_capped(const OrModel* md, int l, const int* topk, const float* g, float I, float xi,
                            int s, float Dhat, float Dbar, float pJ, int last_exec, int cap, OrDecision* out) {
    const int K = md->k, M = md->M, E = md->E;
    OrDecision D;
    std::memset(&D, 0, sizeof(D));
    for (int j = 0; j < K; ++j) { D.topk[j] = topk[j]; D.g[j] = g[j]; }
    D.I = I;
    D.xi = xi;
    D.exit_ok = (l > 0 && last_exec && xi >= pJ) ? 1 : 0;                // Eq. (8), (9), (34)

    // Execute candidates per slot, budget-feasible on their own (Eq. 34).
    std::vector<CandList> cs(K);
    for (int j = 0; j < K; ++j) {
        CandList all = cand_list(md, l, topk[j]);
        for (size_t i = 0; i < all.m.size(); ++i)
            if (Dhat + all.Q[i] <= Dbar) {
                cs[j].m.push_back(all.m[i]); cs[j].k.push_back(all.k[i]); cs[j].Q.push_back(all.Q[i]);
            }
    }
    // Transmission necessity (Eq. 35), summed over slots.
    float Gamma = 0.0f;
    for (int j = 0; j < K; ++j) {
        float gj = kInf;
        for (size_t i = 0; i < cs[j].m.size(); ++i)
            gj = std::min(gj, cs[j].m[i] != s ? md->trans[(size_t)s * M + cs[j].m[i]] : 0.0f);
        Gamma = Gamma + gj;
    }
    D.Gamma = Gamma;
    const float Lambda = md->lambda_[l] * I;                                  // Eq. (5)
    D.Lambda = Lambda;
    D.skip_ok = (Gamma > 0.0f && I <= md->theta[l] && Dhat + Lambda <= Dbar) ? 1 : 0;

    // Look-ahead cost-to-go Phi^{(H-1)}_l (Eq. 39).
    const float R = Dbar - Dhat;
    std::vector<float> phi(M * E);
    or_lookahead_table_capped(md, l, R, Dbar, cap, phi.data());

    // Slot 0: argmin of f + Phi (Eq. 40); later slots: argmin of f.
    float Drun = Dhat;
    float tot = 0.0f;
    for (int j = 0; j < K; ++j) {
        int bi = -1;
        float bv = kInf, bf = 0.0f;
        for (size_t i = 0; i < cs[j].m.size(); ++i) {
            if (!(Drun + cs[j].Q[i] <= Dbar)) continue;
            float f = or_exec_cost(md, l, s, cs[j].m[i], cs[j].Q[i], Dbar);
            float v = (j == 0) ? f + phi[cs[j].m[i] * E + cs[j].k[i]] : f;
            if (bi < 0 || v < bv) { bi = (int)i; bv = v; bf = f; }
        }
        // The exact candidate (Q = 0) is always admissible (Property 2).
        D.exp_sel[j] = cs[j].k[bi];
        D.srv_sel[j] = cs[j].m[bi];
        D.Q_sel[j] = cs[j].Q[bi];
        D.f_sel[j] = bf;
        Drun = Drun + cs[j].Q[bi];
        tot = (j == 0) ? bv : tot + bv;
    }
    D.tot_exec = tot;
    D.tot_skip = kInf;
    if (D.skip_ok) D.tot_skip = md->omega_D * (Lambda / Dbar) + phi[s * E + topk[0]];   // Eq. (32)

    D.action = A_EXEC;
    float best = D.tot_exec;
    if (D.skip_ok && D.tot_skip < D.tot_exec) { D.action = A_SKIP; best = D.tot_skip; }
    if (D.exit_ok && best > 0.0f) D.action = A_EXIT;

    if (D.action == A_EXEC) { D.s_new = D.srv_sel[0]; D.Dhat_new = Drun; }     // Eq. (41)
    else if (D.action == A_SKIP) { D.s_new = s; D.Dhat_new = Dhat + Lambda; }   // Eq. (42)
    else { D.s_new = s; D.Dhat_new = Dhat; }
    D.Lhat = md->N;
    *out = D;
}

void or_decide_given(const OrModel* md, int l, const int* topk, const float* g, float I, float xi,
                     int s, float Dhat, float Dbar, float pJ, int last_exec, OrDecision* out) {
    or_decide_given_capped(md, l, topk, g, I, xi, s, Dhat, Dbar, pJ, last_exec, 1 << 30, out);
}

// Full per-token decision: router + exit head + or_decide_given.
// The router reads h_moe, the input of the MoE sublayer; the exit head of layer
// l-1 and the exit prediction read h_in, the representation entering layer l.
// Without an attention sublayer both are the same state.
void or_decide_token2(const OrModel* md, const OrLayerWeights* lw, int l, const uint16_t* h_moe,
                      const uint16_t* h_in, int s, float Dhat, float Dbar, float pJ, int last_exec,
                      OrDecision* out, float* z_out) {
    std::vector<float> z(md->E), p(md->E);
    int topk[16];
    float g[16], I;
    or_router(md, lw->W_r, lw->b_r, lw->W_norm, h_moe, z.data(), p.data(), topk, g, &I);
    const uint16_t* h = h_in;
    float xi = -1.0f;
    if (l > 0 && last_exec && lw->W_x_prev)
        xi = or_exit_conf(md, lw->W_x_prev, lw->b_x_prev, h, lw->W_norm != nullptr, nullptr);
    // Predicted exit layer (Eq. 36) caps the look-ahead: layers >= L_hat are
    // predicted not to run, so they add no cost-to-go.
    int Lhat = md->N, cap = 1 << 30;
    float cgap = kInf, cbest = 0.0f;
    if (md->n_centroids > 0 && lw->centroids) {
        Lhat = or_predict_exit(md, lw->centroids, lw->centroid_exit, h, &cbest, &cgap);
        cap = Lhat - 1 - l;
    }
    or_decide_given_capped(md, l, topk, g, I, xi, s, Dhat, Dbar, pJ, last_exec, cap, out);
    out->Lhat = Lhat;
    // Near-threshold flags for the comparison protocol.
    const float band = 1e-5f;
    int nr = 0;
    if (cgap <= band * std::max(1.0f, std::fabs(cbest))) nr |= 32;
    if (std::fabs(I - md->theta[l]) <= band) nr |= 1;
    if (xi >= 0.0f && std::fabs(xi - pJ) <= band) nr |= 2;
    {
        std::vector<float> zs(z);
        std::sort(zs.begin(), zs.end(), std::greater<float>());
        int lim = std::min(md->k + 1, md->E);
        for (int j = 0; j + 1 < lim; ++j)
            if (zs[j] - zs[j + 1] <= band) nr |= 4;
    }
    if (std::fabs(Dhat + out->Lambda - Dbar) <= band) nr |= 8;
    if (out->skip_ok) {
        float mn = std::min(out->tot_exec, out->tot_skip);
        if (std::fabs(out->tot_skip - out->tot_exec) <= band * std::max(1.0f, std::fabs(mn))) nr |= 16;
    }
    out->near = nr;
    if (z_out) for (int e = 0; e < md->E; ++e) z_out[e] = z[e];
}

void or_decide_token(const OrModel* md, const OrLayerWeights* lw, int l, const uint16_t* h, int s,
                     float Dhat, float Dbar, float pJ, int last_exec, OrDecision* out, float* z_out) {
    or_decide_token2(md, lw, l, h, h, s, Dhat, Dbar, pJ, last_exec, out, z_out);
}

// ------------------------------------------------------- attention sublayer
//
// The paper keeps attention local to the token's server and treats it as a fixed
// per-layer term (Sec. III-C, attention placement): a skip bypasses only the FFN
// sublayer, the attention sublayer still runs.  Its arithmetic follows the
// model families of Sec. VI-A (pre-norm transformer blocks): RMSNorm, rotary
// position embedding, grouped-query causal softmax attention, output projection
// with the residual.

// Rotary position embedding of one head vector of length Dh: element i pairs
// with i + Dh/2 and turns by the angle pos * theta^(-2i/Dh).
void or_rope(const double* x, int Dh, int pos, double theta, double* y) {
    const int half = Dh / 2;
    for (int i = 0; i < half; ++i) {
        const double ang = (double)pos * std::pow(theta, -2.0 * i / Dh);
        const double c = std::cos(ang), sn = std::sin(ang);
        y[i] = x[i] * c - x[i + half] * sn;
        y[i + half] = x[i + half] * c + x[i] * sn;
    }
}

// h_mid = h + attention(h) for the live tokens with row_mask set (every live
// token when row_mask is NULL); all other rows of h_mid are copies of h.
//   a = bf16(h * r * gamma)                        (r: RMS factor of h)
//   q = bf16(rope(a W_q^T, pos)), k = bf16(rope(a W_k^T, pos)) per head,
//   v = bf16(a W_v^T)                               pos = t mod S
//   o_head = bf16( sum_j softmax_j(q . k_j / sqrt(Dh)) v_j )
//            over the tokens j of t's sequence (t - pos .. t), query head
//            hq reading key/value head hq / (Hq / Hkv)
//   h_mid = bf16(h + o W_o^T)
// Keys and values come from every token of the sequence, live or not: a token
// that left keeps its last state, which later tokens still attend to.
int or_attention(const OrModel* md, const OrLayerWeights* lw, int T, const uint16_t* h, const uint8_t* alive,
                 const uint8_t* row_mask, uint16_t* h_mid, int nthreads) {
    const int d = md->d, Hq = md->attn_heads, Hkv = md->attn_kv_heads, Dh = md->head_dim, S = md->attn_seq;
    if (Hq <= 0 || Hkv <= 0 || Hq % Hkv || Dh <= 0 || Dh % 2 || S <= 0 || !lw->W_qkv || !lw->W_o ||
        !lw->W_attn_norm)
        return -1;
    const int nq = Hq * Dh, nkv = Hkv * Dh, nqkv = nq + 2 * nkv, grp = Hq / Hkv;
    std::memcpy(h_mid, h, (size_t)T * d * sizeof(uint16_t));
    std::vector<char> query(T, 0), need(T, 0);
    for (int t = 0; t < T; ++t) {
        if (!alive[t] || (row_mask && !row_mask[t])) continue;
        query[t] = 1;
        for (int j = t - t % S; j <= t; ++j) need[j] = 1;
    }
    // Projections of the tokens needed, RoPE on query and key heads.
    std::vector<uint16_t> qkv((size_t)T * nqkv, 0);
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 4)
#endif
    for (int t = 0; t < T; ++t) {
        if (!need[t]) continue;
        const uint16_t* hr = h + (size_t)t * d;
        const double r = or_rms_factor(hr, d, md->norm_eps);
        std::vector<uint16_t> a(d);
        for (int i = 0; i < d; ++i) a[i] = d2bf((double)bf2f(hr[i]) * r * (double)bf2f(lw->W_attn_norm[i]));
        std::vector<double> z(nqkv);
        for (int o = 0; o < nqkv; ++o) z[o] = dot_bf16(a.data(), lw->W_qkv + (size_t)o * d, d);
        const int pos = t % S;
        std::vector<double> y(Dh);
        for (int hh = 0; hh < Hq + Hkv; ++hh) {          // query heads, then key heads
            or_rope(z.data() + (size_t)hh * Dh, Dh, pos, (double)md->rope_theta, y.data());
            std::copy(y.begin(), y.end(), z.begin() + (size_t)hh * Dh);
        }
        uint16_t* out = qkv.data() + (size_t)t * nqkv;
        for (int o = 0; o < nqkv; ++o) out[o] = d2bf(z[o]);
    }
    const double scale = 1.0 / std::sqrt((double)Dh);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 4)
#endif
    for (int t = 0; t < T; ++t) {
        if (!query[t]) continue;
        const int j0 = t - t % S;
        const uint16_t* qt = qkv.data() + (size_t)t * nqkv;
        std::vector<uint16_t> o(nq);
        std::vector<double> w(t - j0 + 1), acc(Dh);
        for (int hq = 0; hq < Hq; ++hq) {
            const int g = hq / grp;
            double mx = -std::numeric_limits<double>::infinity();
            for (int j = j0; j <= t; ++j) {
                const uint16_t* kj = qkv.data() + (size_t)j * nqkv + nq + (size_t)g * Dh;
                w[j - j0] = dot_bf16(qt + (size_t)hq * Dh, kj, Dh) * scale;
                mx = std::max(mx, w[j - j0]);
            }
            double den = 0.0;
            for (int j = j0; j <= t; ++j) { w[j - j0] = std::exp(w[j - j0] - mx); den += w[j - j0]; }
            std::fill(acc.begin(), acc.end(), 0.0);
            for (int j = j0; j <= t; ++j) {
                const uint16_t* vj = qkv.data() + (size_t)j * nqkv + nq + nkv + (size_t)g * Dh;
                for (int i = 0; i < Dh; ++i) acc[i] += w[j - j0] / den * (double)bf2f(vj[i]);
            }
            for (int i = 0; i < Dh; ++i) o[(size_t)hq * Dh + i] = d2bf(acc[i]);
        }
        const uint16_t* hr = h + (size_t)t * d;
        for (int c = 0; c < d; ++c)
            h_mid[(size_t)t * d + c] = d2bf((double)bf2f(hr[c]) + dot_bf16(o.data(), lw->W_o + (size_t)c * nq, nq));
    }
    return 0;
}

// ------------------------------------------------------------- expert FFN

// One expert on one row: act = silu(x W1^T) * (x W3^T) (SwiGLU) or relu(x W1^T),
// rounded to bf16; y = act W2^T rounded to bf16.  Dot products in double.
void or_ffn_row(int d, int F, int act, const uint16_t* W13, const uint16_t* W2, const uint16_t* x,
                uint16_t* y) {
    std::vector<double> a(F);
    for (int c = 0; c < F; ++c) {
        double v;
        if (act == 1) {
            int gr = (c / kGateUpGroup) * 2 * kGateUpGroup + (c % kGateUpGroup);
            double gt = dot_bf16(x, W13 + (size_t)gr * d, d);
            double up = dot_bf16(x, W13 + (size_t)(gr + kGateUpGroup) * d, d);
            v = gt / (1.0 + std::exp(-gt)) * up;
        } else {
            v = std::max(0.0, dot_bf16(x, W13 + (size_t)c * d, d));
        }
        a[c] = (double)bf2f(d2bf(v));
    }
    for (int o = 0; o < d; ++o) {
        const uint16_t* w = W2 + (size_t)o * F;
        double acc = 0.0;
        for (int c = 0; c < F; ++c) acc += a[c] * (double)bf2f(w[c]);
        y[o] = d2bf(acc);
    }
}

// ---------------------------------------------------------------- layer step

// One MoE layer over T tokens (the per-layer body of Algorithm 2 plus the MoE computation the
// decisions gate).  h is bf16 [T][d], updated in place.  row_mask (may be NULL)
// limits the FFN/combine to the selected tokens; decisions, state and
// compaction are always computed for every token.
//
// With an attention sublayer (md->attn_heads > 0) the layer is the full block:
// h_mid = h + attention(h) for the live tokens (computed here when h_mid_in is
// NULL, else taken from h_mid_in), the router, the experts and the residual read
// h_mid, the exit head reads h; executed and skipped tokens leave with
// h_mid + FFN (h_mid alone for a skip without a shared expert), while a token
// that exits at this layer keeps h (layers from l on do not run for it).
int or_layer_step_block(const OrModel* md, const OrLayerWeights* lw, int l, int T, uint16_t* h,
                        const uint16_t* h_mid_in, OrTokens* tk, OrLayerOut* out, const uint8_t* row_mask,
                        int nthreads) {
    const int K = md->k, E = md->E, d = md->d;
    if (l < 0 || l >= md->N || T < 0) return -1;
    const bool block = md->attn_heads > 0;
    std::vector<uint16_t> hmid;
    if (block) {
        hmid.resize((size_t)T * d);
        if (h_mid_in) std::memcpy(hmid.data(), h_mid_in, (size_t)T * d * sizeof(uint16_t));
        else if (or_attention(md, lw, T, h, tk->alive, nullptr, hmid.data(), nthreads)) return -1;
    }
    const uint16_t* hm = block ? hmid.data() : h;
    std::vector<OrDecision> dec(T);
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 4)
#endif
    for (int t = 0; t < T; ++t) {
        OrDecision& D = dec[t];
        if (!tk->alive[t]) { std::memset(&D, 0, sizeof(D)); D.action = A_DEAD; D.xi = -1.0f; continue; }
        or_decide_token2(md, lw, l, hm + (size_t)t * d, h + (size_t)t * d, tk->s[t], tk->Dhat[t], tk->Dbar[t],
                         tk->pJ[t], tk->last_exec[t], &D, nullptr);
    }
    // Compaction: executed (token, slot) pairs stably ordered by expert, then
    // the tokens that run the shared expert (executed or skipped), by token.
    std::vector<std::pair<int, int>> pairs;   // (expert, t*K + j)
    for (int t = 0; t < T; ++t)
        if (dec[t].action == A_EXEC)
            for (int j = 0; j < K; ++j) pairs.push_back({dec[t].exp_sel[j], t * K + j});
    std::stable_sort(pairs.begin(), pairs.end(),
                     [](const std::pair<int, int>& a, const std::pair<int, int>& b) { return a.first < b.first; });
    std::vector<int> shared_rows;
    if (md->F_sh > 0)
        for (int t = 0; t < T; ++t)
            if (dec[t].action == A_EXEC || dec[t].action == A_SKIP) shared_rows.push_back(t);
    std::vector<int> goff(E + 2, 0);
    for (auto& pr : pairs) goff[pr.first + 1]++;
    for (int e = 0; e < E; ++e) goff[e + 1] += goff[e];
    goff[E + 1] = goff[E] + (int)shared_rows.size();
    std::vector<int> pos((size_t)T * K, -1), pos_sh(T, -1);
    for (size_t p = 0; p < pairs.size(); ++p) pos[pairs[p].second] = (int)p;
    for (size_t i = 0; i < shared_rows.size(); ++i) pos_sh[shared_rows[i]] = (int)i;

    // Expert FFN on selected rows, then the gate-weighted combine with residual.
    std::vector<uint16_t> hin(hm, hm + (size_t)T * d);
#ifdef _OPENMP
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int t = 0; t < T; ++t) {
        const OrDecision& D = dec[t];
        if (D.action != A_EXEC && D.action != A_SKIP) continue;
        if (row_mask && !row_mask[t]) continue;
        const uint16_t* hrow = hin.data() + (size_t)t * d;
        std::vector<float> acc(d);
        for (int o = 0; o < d; ++o) acc[o] = bf2f(hrow[o]);
        // Expert input: bf16 rounding of the normalised state (or h itself).
        std::vector<uint16_t> xn(hrow, hrow + d);
        if (lw->W_norm) {
            const double r = or_rms_factor(hrow, d, md->norm_eps);
            for (int i = 0; i < d; ++i) xn[i] = d2bf((double)bf2f(hrow[i]) * r * (double)bf2f(lw->W_norm[i]));
        }
        const uint16_t* x = xn.data();
        std::vector<uint16_t> y(d);
        if (D.action == A_EXEC) {
            float gs = 0.0f;
            for (int j = 0; j < K; ++j) gs = gs + D.g[j];
            const size_t n13 = (md->act == 1) ? 2 : 1;
            for (int j = 0; j < K; ++j) {
                int e = D.exp_sel[j];
                or_ffn_row(d, md->F, md->act, lw->W13 + (size_t)e * n13 * md->F * d,
                           lw->W2 + (size_t)e * d * md->F, x, y.data());
                float gw = md->renorm_topk ? D.g[j] / gs : D.g[j];
                for (int o = 0; o < d; ++o) acc[o] = acc[o] + gw * bf2f(y[o]);
            }
        }
        if (md->F_sh > 0) {
            or_ffn_row(d, md->F_sh, 1, lw->W13_sh, lw->W2_sh, x, y.data());
            for (int o = 0; o < d; ++o) acc[o] = acc[o] + bf2f(y[o]);
        }
        for (int o = 0; o < d; ++o) h[(size_t)t * d + o] = f2bf(acc[o]);
    }

    // State update (Eq. 41, 42 and exit) and outputs.
    for (int t = 0; t < T; ++t) {
        const OrDecision& D = dec[t];
        if (out) {
            if (out->action) out->action[t] = (uint8_t)D.action;
            if (out->xi) out->xi[t] = D.xi;
            if (out->I) out->I[t] = D.action == A_DEAD ? 0.0f : D.I;
            if (out->near) out->near[t] = (uint8_t)D.near;
            if (out->Gamma) out->Gamma[t] = D.Gamma;
            if (out->tot_exec) out->tot_exec[t] = D.tot_exec;
            if (out->tot_skip) out->tot_skip[t] = D.tot_skip;
            if (out->lhat) out->lhat[t] = (int16_t)(D.action == A_DEAD ? -1 : D.Lhat);
            for (int j = 0; j < K; ++j) {
                if (out->topk_idx) out->topk_idx[t * K + j] = D.action == A_DEAD ? -1 : D.topk[j];
                if (out->topk_g) out->topk_g[t * K + j] = D.action == A_DEAD ? 0.0f : D.g[j];
                if (out->exp_sel) out->exp_sel[t * K + j] = D.action == A_EXEC ? (uint8_t)D.exp_sel[j] : 0xFF;
                if (out->srv_sel) out->srv_sel[t * K + j] = D.action == A_EXEC ? (uint8_t)D.srv_sel[j] : 0xFF;
            }
        }
        if (D.action == A_DEAD) continue;
        if (D.xi >= 0.0f) tk->xi_last[t] = D.xi;
        if (D.action == A_EXEC) { tk->s[t] = (uint8_t)D.s_new; tk->Dhat[t] = D.Dhat_new; tk->last_exec[t] = 1; }
        else if (D.action == A_SKIP) { tk->Dhat[t] = D.Dhat_new; tk->last_exec[t] = 0; }
        else { tk->alive[t] = 0; tk->exit_layer[t] = (int16_t)l; }
    }
    if (out && out->perm) {
        for (size_t p = 0; p < pairs.size(); ++p) out->perm[p] = pairs[p].second;
        for (size_t i = 0; i < shared_rows.size(); ++i) out->perm[pairs.size() + i] = shared_rows[i];
    }
    if (out && out->group_off) for (int e = 0; e < E + 2; ++e) out->group_off[e] = goff[e];
    return 0;
}

int or_layer_step(const OrModel* md, const OrLayerWeights* lw, int l, int T, uint16_t* h,
                  OrTokens* tk, OrLayerOut* out, const uint8_t* row_mask, int nthreads) {
    return or_layer_step_block(md, lw, l, T, h, nullptr, tk, out, row_mask, nthreads);
}

// Whole forward: layers 0..N-1 (the layer loop of Algorithm 2).
int or_forward(const OrModel* md, const OrLayerWeights* lws, int T, uint16_t* h, OrTokens* tk,
               int nthreads) {
    for (int l = 0; l < md->N; ++l) {
        int rc = or_layer_step_block(md, &lws[l], l, T, h, nullptr, tk, nullptr, nullptr, nthreads);
        if (rc) return rc;
    }
    return 0;
}

// ------------------------------------------------------- runtime feedback

typedef struct {
    int user_size;      // tokens per user (consecutive blocks)
    float eta;          // step of Eq. (37)
    float p_min;        // floor of the projection in Eq. (37)
    float kappa;        // step of Eq. (43)
} OrFeedbackCfg;

typedef struct {
    float omega_T, omega_D;
    double T_norm, D_util;
    int users_updated;
} OrFeedbackOut;

// Feedback at the end of an observation window (the periodic update of Algorithm 2).
// Eq. (37): for every user with exits in the window, p_J <- clamp(p_J +
// eta * (xi_exit_mean - p_J), p_min, 1), where xi_exit_mean is the mean exit
// confidence of the user's exited tokens.  Eq. (43): omega_D <- clamp(omega_D
// + kappa * (D_util - T_norm), 0, 1), omega_T = 1 - omega_D, where D_util is the
// mean over users of sum(Dhat) / sum(Dbar) and T_norm is the window's summed
// per-step delay over its full-depth exact reference (ref_slots * d_ref).
int or_feedback(const OrFeedbackCfg* fb, int T, int N, float* pJ, const uint8_t* alive,
                const int16_t* exit_layer, const float* xi_last, const float* Dhat, const float* Dbar,
                double delay_sum_ms, double ref_slots, float d_ref, float omega_D, OrFeedbackOut* out) {
    if (!fb || fb->user_size < 1 || T < 0) return -1;
    const int us = fb->user_size;
    const int users = (T + us - 1) / us;
    double util_sum = 0.0;
    int updated = 0;
    for (int u = 0; u < users; ++u) {
        const int t0 = u * us, t1 = std::min(T, t0 + us);
        double xs = 0.0, dh = 0.0, db = 0.0;
        int n = 0;
        for (int t = t0; t < t1; ++t) {
            if (!alive[t] && exit_layer[t] < N) { xs += (double)xi_last[t]; ++n; }
            dh += (double)Dhat[t];
            db += (double)Dbar[t];
        }
        if (n > 0) {
            const float xbar = (float)(xs / n);
            for (int t = t0; t < t1; ++t) {
                float q = pJ[t] + fb->eta * (xbar - pJ[t]);
                q = std::min(std::max(q, fb->p_min), 1.0f);
                pJ[t] = q;
            }
            ++updated;
        }
        util_sum += (db > 0.0) ? dh / db : 0.0;
    }
    const double D_util = users > 0 ? util_sum / users : 0.0;
    const double T_norm = (ref_slots > 0.0) ? delay_sum_ms / (ref_slots * (double)d_ref) : 0.0;
    double wD = (double)omega_D + (double)fb->kappa * (D_util - T_norm);
    wD = std::min(std::max(wD, 0.0), 1.0);
    out->omega_D = (float)wD;
    out->omega_T = 1.0f - out->omega_D;
    out->T_norm = T_norm;
    out->D_util = D_util;
    out->users_updated = updated;
    return 0;
}

// ------------------------------------------------- offline stage (Algorithm 1)

// Calibration counts of one layer from its decisions (Algorithm 1, statistics
// behind Eq. 26-28 and 38).  For every token live at layer l: one active count
// (pi_l), one residence count on its server before the layer (rho_{m,l}), one
// activation count per routed slot (a_l^k), one above-threshold count per slot
// when I > theta_l (sigma_l^k); and, when the token was live at l-1 too, one
// transition count from its slot-0 target at l-1 to its slot-0 target at l
// (Eq. 38).  prev_target[t] carries the slot-0 target between layers (-1 none).
int or_calib_accumulate(const OrModel* md, int l, int T, const int32_t* topk_idx, const float* I,
                        const uint8_t* action, const uint8_t* s_before, int16_t* prev_target,
                        uint64_t* c_trans, uint64_t* c_alive, uint64_t* c_resid, uint64_t* c_act,
                        uint64_t* c_above) {
    const int E = md->E, K = md->k, M = md->M;
    for (int t = 0; t < T; ++t) {
        if (action[t] == A_DEAD) continue;
        c_alive[l] += 1;
        c_resid[(size_t)l * M + s_before[t]] += 1;
        for (int j = 0; j < K; ++j) {
            const int r = topk_idx[t * K + j];
            c_act[(size_t)l * E + r] += 1;
            if (I[t] > md->theta[l]) c_above[(size_t)l * E + r] += 1;
        }
        const int r0 = topk_idx[t * K];
        if (l > 0 && prev_target[t] >= 0) c_trans[((size_t)(l - 1) * E + prev_target[t]) * E + r0] += 1;
        prev_target[t] = (int16_t)r0;
    }
    return 0;
}

// Offline statistics from the counts over T_cal calibration tokens:
// P_l(k -> k') = n_l(k -> k') / sum_k'' n_l(k -> k'') (Eq. 38; a row without
// observations stays uniform), pi_l = active_l / T_cal (Eq. 26),
// sigma_l^k = above_l^k / routed_l^k (Eq. 27; 0 without observations),
// a_l^k = routed_l^k / (k * active_l), lambda_l^k = pi_l sigma_l^k a_l^k,
// rho_{m,l} = resident_{m,l} / active_l.
int or_calib_finalize(const OrModel* md, long long T_cal, const uint64_t* c_trans, const uint64_t* c_alive,
                      const uint64_t* c_resid, const uint64_t* c_act, const uint64_t* c_above, float* P,
                      float* pi, float* sigma, float* act, float* lam, float* rho) {
    const int N = md->N, E = md->E, M = md->M, K = md->k;
    for (int l = 0; l + 1 < N; ++l)
        for (int k = 0; k < E; ++k) {
            uint64_t tot = 0;
            for (int kp = 0; kp < E; ++kp) tot += c_trans[((size_t)l * E + k) * E + kp];
            for (int kp = 0; kp < E; ++kp)
                P[((size_t)l * E + k) * E + kp] =
                    tot ? (float)((double)c_trans[((size_t)l * E + k) * E + kp] / (double)tot) : (float)(1.0 / E);
        }
    for (int l = 0; l < N; ++l) {
        const double a = (double)c_alive[l];
        pi[l] = T_cal > 0 ? (float)(a / (double)T_cal) : 0.0f;
        for (int k = 0; k < E; ++k) {
            const double routed = (double)c_act[(size_t)l * E + k];
            sigma[(size_t)l * E + k] = routed > 0 ? (float)((double)c_above[(size_t)l * E + k] / routed) : 0.0f;
            act[(size_t)l * E + k] = a > 0 ? (float)(routed / (K * a)) : 0.0f;
            lam[(size_t)l * E + k] = pi[l] * sigma[(size_t)l * E + k] * act[(size_t)l * E + k];
        }
        for (int m = 0; m < M; ++m) rho[(size_t)l * M + m] = a > 0 ? (float)((double)c_resid[(size_t)l * M + m] / a) : 0.0f;
    }
    return 0;
}

// Greedy communication-aware replication (Algorithm 1, Eq. 28, (c.1)-(c.3)).
// Benefit of a replica of expert k of layer l on server m that does not hold
// it: B = lambda_l^k * rho_{m,l} * mean over the servers m' holding it of
// trans[m][m'] (the combined z/B + tau delay from m).  Each iteration evaluates
// every feasible pair (not yet placed, fits the residual memory of m), places
// the largest benefit (ties: lowest (m, l, k) in that order) and updates the
// residual memory; it stops when no feasible pair remains.  place is updated
// in place; returns the number of replicas added.
int or_replicate(const OrModel* md, const float* lam, const float* rho, const double* expert_bytes,
                 const double* capacity, uint16_t* place) {
    const int N = md->N, E = md->E, M = md->M;
    std::vector<double> used(M, 0.0);
    for (int l = 0; l < N; ++l)
        for (int k = 0; k < E; ++k)
            for (int m = 0; m < M; ++m)
                if ((place[(size_t)l * E + k] >> m) & 1u) used[m] += expert_bytes[(size_t)l * E + k];
    int added = 0;
    while (true) {
        double best = -1.0;
        int bm = -1, bl = -1, bk = -1;
        for (int m = 0; m < M; ++m)
            for (int l = 0; l < N; ++l)
                for (int k = 0; k < E; ++k) {
                    const uint16_t mask = place[(size_t)l * E + k];
                    if ((mask >> m) & 1u) continue;
                    if (used[m] + expert_bytes[(size_t)l * E + k] > capacity[m]) continue;
                    double dsum = 0.0;
                    int hosts = 0;
                    for (int mp = 0; mp < M; ++mp)
                        if ((mask >> mp) & 1u) { dsum += (double)md->trans[(size_t)m * M + mp]; ++hosts; }
                    const double reach = hosts ? dsum / hosts : 0.0;
                    const double B = (double)lam[(size_t)l * E + k] * (double)rho[(size_t)l * M + m] * reach;
                    if (B > best) { best = B; bm = m; bl = l; bk = k; }
                }
        if (bm < 0) break;
        place[(size_t)bl * E + bk] |= (uint16_t)(1u << bm);
        used[bm] += expert_bytes[(size_t)bl * E + bk];
        ++added;
    }
    return added;
}

int or_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

}  // extern "C"
