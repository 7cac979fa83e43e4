// Kernel (a): exit gate + skip test + substitute-or-fetch with server argmin and
// look-ahead + state update, one group of 8, 16 or 32 lanes per live token (the
// smallest group with a lane per expert).
//
// Paper: Sec. V, the per-token body of Algorithm 2.  Router and importance: Eq. (4);
// exit confidence: Eq. (7)-(9); skip admission: Eq. (5), (34), (35); per-step
// cost: Eq. (30)-(32); look-ahead cost-to-go: Eq. (38)-(39); choice: Eq. (40);
// updates: Eq. (41)-(42).
//
// The router and exit-head logits come from kernel a0 (router.cu).  Every
// decision quantity after them is fp32 with one fixed operation order written
// with explicit round-to-nearest intrinsics (no fused multiply-add), so that the
// integer outcomes are reproducible bit for bit.  The delay part of the execute
// cost, omega_T * (d / d_ref), is read from a per-layer table computed at create
// with the same operations.
//
// Look-ahead per future layer l': (1) one pass over the layer's candidates
// stages, in shared memory, the feasibility (Q <= R), the quality term
// omega_D * Q / Dbar and the deeper cost-to-go Phi(m_c, k_c) of each
// candidate; (2) each (m, k') value is a minimum over its candidates of
// table + staged terms; (3) Phi_{l'-1}(m, k) = sum_k' P(k -> k') V(m, k').
#include <float.h>

#include "internal.cuh"

namespace tmoe {

namespace {

constexpr int kWarps = 4;
#define kInf __int_as_float(0x7f800000)

// Reductions over the G lanes of one token's group (mask gmask); arg-reductions
// break ties to the lower index.
template <int G>
__device__ __forceinline__ float grp_sum(unsigned gmask, float v) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) v += __shfl_xor_sync(gmask, v, o);
    return v;
}
template <int G>
__device__ __forceinline__ float grp_max(unsigned gmask, float v) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(gmask, v, o));
    return v;
}
template <int G>
__device__ __forceinline__ float grp_min(unsigned gmask, float v) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) v = fminf(v, __shfl_xor_sync(gmask, v, o));
    return v;
}
template <int G>
__device__ __forceinline__ void grp_argmin(unsigned gmask, float& v, int& i) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) {
        float ov = __shfl_xor_sync(gmask, v, o);
        int oi = __shfl_xor_sync(gmask, i, o);
        if (ov < v || (ov == v && oi < i)) { v = ov; i = oi; }
    }
}
template <int G>
__device__ __forceinline__ void grp_argmax(unsigned gmask, float& v, int& i) {
#pragma unroll
    for (int o = G / 2; o > 0; o >>= 1) {
        float ov = __shfl_xor_sync(gmask, v, o);
        int oi = __shfl_xor_sync(gmask, i, o);
        if (ov > v || (ov == v && oi < i)) { v = ov; i = oi; }
    }
}

// Sum of n partial sums base[0], base[stride], ... added in index order.  The
// loads of a batch of eight are issued before the additions, so a token's
// column ranges cost one memory latency per batch rather than one each (the
// order of the additions, and so the result, is unchanged).
__device__ __forceinline__ float sum_parts(const float* __restrict__ base, size_t stride, int n) {
    float acc = 0.f;
    int i = 0;
    for (; i + 8 <= n; i += 8) {
        float v[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) v[u] = base[(size_t)(i + u) * stride];
#pragma unroll
        for (int u = 0; u < 8; ++u) acc = __fadd_rn(acc, v[u]);
    }
    for (; i < n; ++i) acc = __fadd_rn(acc, base[(size_t)i * stride]);
    return acc;
}

// The same for up to kMS values at once: value u sums base[off + u * ustride]
// over the n parts (u < nv), parts in index order.  Every load of one part is
// issued before the additions.
constexpr int kMS = 8;
__device__ __forceinline__ void multi_sum(const float* __restrict__ base, size_t stride, int n, int off,
                                          int ustride, int nv, float (&out)[kMS]) {
#pragma unroll
    for (int u = 0; u < kMS; ++u) out[u] = 0.f;
    if (nv == 1) {
        out[0] = sum_parts(base + off, stride, n);
        return;
    }
    for (int i = 0; i < n; ++i) {
        float v[kMS];
#pragma unroll
        for (int u = 0; u < kMS; ++u) v[u] = u < nv ? base[(size_t)i * stride + off + u * ustride] : 0.f;
#pragma unroll
        for (int u = 0; u < kMS; ++u) out[u] = __fadd_rn(out[u], v[u]);
    }
}

struct WarpCounters {
    unsigned long long layer_tokens, exec_tokens, skipped, exited;
    unsigned long long le, ls, re, rs, hops, shared_phi;
    float delay;          // this warp's tokens (a handful): fp32 is enough for the statistic
    float max_ratio;
};

// G lanes per token (8, 16 or 32): a warp decides 32 / G tokens at once.  With
// E <= G every per-expert value sits in its own lane, so the reduction trees
// over experts are those of a full warp with the unused lanes at zero.
// Seven blocks per SM (72 registers, a few bytes spilled): each token is a
// chain of dependent reads, so warps in flight matter more than registers
// (six blocks at 80 registers: 1.31 instead of 0.94 ms per Mixtral-shaped
// forward, 1.59 instead of 1.45 ms per Qwen-shaped one).
template <int G>
__global__ void __launch_bounds__(kWarps * 32, 7) decide_kernel(const DecideParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    extern __shared__ float smem[];
    const int lane = threadIdx.x & (G - 1);          // lane within the token's group
    const int warp = threadIdx.x >> 5;
    const int grp = (threadIdx.x & 31) / G;
    const unsigned gmask = G == 32 ? 0xffffffffu : (((1u << G) - 1u) << (grp * G));
    constexpr int kGroups = kWarps * (32 / G);      // tokens in flight per block
    const int slot = warp * (32 / G) + grp;
    const int E = p.E, M = p.M, C = p.C, K = p.k, l = p.layer;
    const int ME = M * E;
    const int MC = p.tab.max_layer_cand;
    // Per-group scratch: logits z[E], probabilities pr[E], head logits x[C]
    // in shared memory; look-ahead tables V[M*E] and Phi[M*E] and the staged
    // candidate terms after them, or in the group's global slot.
    const size_t per_head = (size_t)(2 * E + C);
    const size_t per_la = (size_t)(2 * ME + 2 * MC) + (size_t)((MC + 3) / 4) * 2;
    float* zs = smem + (size_t)slot * (p.la_scratch ? per_head : per_head + per_la);
    float* ps = zs + E;
    float* xs = ps + E;
    float* bufV = p.la_scratch ? p.la_scratch + ((size_t)blockIdx.x * kGroups + slot) * per_la : xs + C;
    float* bufPhi = bufV + ME;
    float* cqt = bufPhi + ME;                  // omega_D * Q / Dbar, or -1: no quality term
    float* cph = cqt + MC;                     // deeper cost-to-go of the candidate
    uint8_t* cok = reinterpret_cast<uint8_t*>(cph + MC);   // Q <= R
    uint8_t* cmv = cok + ((MC + 3) & ~3);                  // server of the candidate

    __shared__ unsigned long long blk_cnt[10];
    __shared__ double blk_delay;
    __shared__ unsigned int blk_ratio;
    if (threadIdx.x < 10) blk_cnt[threadIdx.x] = 0ull;
    if (threadIdx.x == 0) { blk_delay = 0.0; blk_ratio = 0u; }
    __syncthreads();

    const int* coff_l = p.tab.cand_off + l * (E + 1);
    const float* ct_l = p.tab.ctab + (size_t)l * M * M;

    WarpCounters wc = {};
    const int ngroups = gridDim.x * kGroups;
    for (int t = blockIdx.x * kGroups + slot; t < p.T; t += ngroups) {
        // The token's state is read before the liveness test: the loads overlap.
        const int alive_t = p.alive[t];
        const int s = p.s[t];
        const float Dhat = p.Dhat[t];
        const float Dbar = p.Dbar[t];
        const float pJ = p.pJ[t];
        const int last_exec = p.last_exec[t];
        if (!alive_t) {
            if (lane == 0) {
                p.action[t] = 3;
                p.I_out[t] = 0.f;
                p.xi_out[t] = -1.f;
                if (p.lhat_out) p.lhat_out[t] = -1;
            }
            if (lane < K) {
                p.topk_idx[t * K + lane] = -1;
                p.topk_g[t * K + lane] = 0.f;
                p.exp_sel[t * K + lane] = 0xFF;
                p.srv_sel[t * K + lane] = 0xFF;
            }
            continue;
        }

        // Router logits: partial dot products of kernel a0 summed over the column
        // ranges in order, times the RMS factor, plus the bias; softmax (Eq. 4),
        // top-k by logit (a NaN logit ranks as -infinity).
        float rn = 1.f;
        const size_t kstride = (size_t)p.zs;      // the column ranges of a token are contiguous
        const float* zrow = p.zpart + (size_t)t * p.ksplit * p.zs;
        float zacc = lane < E ? sum_parts(zrow + lane, kstride, p.ksplit) : 0.f;
        if (p.use_norm) {
            const float sq = sum_parts(p.sqpart + (size_t)t * p.ksplit, 1, p.ksplit);
            rn = rsqrtf(sq / (float)p.d + p.norm_eps);
            if (lane == 0) p.rnorm[t] = rn;
        }
        for (int e = lane; e < E; e += G) {
            const float acc = e == lane ? zacc : sum_parts(zrow + e, kstride, p.ksplit);
            const float v = __fadd_rn(__fmul_rn(acc, rn), p.bias[e]);
            zs[e] = (v != v) ? -kInf : v;
        }
        __syncwarp(gmask);
        float zmax = -FLT_MAX;
        for (int e = lane; e < E; e += G) zmax = fmaxf(zmax, zs[e]);
        zmax = grp_max<G>(gmask, zmax);
        float S = 0.f;
        for (int e = lane; e < E; e += G) {
            const float ex = expf(zs[e] - zmax);
            ps[e] = ex;
            S += ex;
        }
        S = grp_sum<G>(gmask, S);
        __syncwarp(gmask);
        for (int e = lane; e < E; e += G) ps[e] = __fdiv_rn(ps[e], S);
        __syncwarp(gmask);
        int topk[kMaxK];
        float g[kMaxK];
        unsigned used = 0u;   // bit i: expert lane + G i taken
        for (int j = 0; j < K; ++j) {
            float bz = -kInf;
            int be = 0x7fffffff;
            for (int i = 0, e = lane; e < E; ++i, e += G)
                if (!((used >> i) & 1u) && (zs[e] > bz || (zs[e] == bz && e < be))) { bz = zs[e]; be = e; }
            grp_argmax<G>(gmask, bz, be);
            topk[j] = be;
            if ((be % G) == lane) used |= 1u << (be / G);
        }
        float I = 0.f;
        for (int j = 0; j < K; ++j) { g[j] = ps[topk[j]]; I = __fadd_rn(I, g[j]); }

        // Exit confidence of the previous layer's head (Eq. 7), exit gate (Eq. 8-9).
        float xi = -1.f;
        const bool have_xi = (l > 0) && last_exec && p.has_head;
        if (have_xi) {
            // The exit head reads the state entering the layer; with an attention
            // sublayer in front of the MoE step that state has its own RMS factor.
            float rx = rn;
            if (p.use_norm && p.sqpart_x) {
                const float sq = sum_parts(p.sqpart_x + (size_t)t * p.ksplit, 1, p.ksplit);
                rx = rsqrtf(sq / (float)p.d + p.norm_eps);
            }
            // This lane's classes c = lane + G u, kMS at a time.
            for (int c0 = lane; c0 < C; c0 += kMS * G) {
                const int nv = min(kMS, (C - c0 + G - 1) / G);
                float acc[kMS];
                multi_sum(zrow, kstride, p.ksplit, E + c0, G, nv, acc);
#pragma unroll
                for (int u = 0; u < kMS; ++u)
                    if (u < nv) xs[c0 + u * G] = __fadd_rn(__fmul_rn(acc[u], rx), p.bias[E + c0 + u * G]);
            }
            __syncwarp(gmask);
            if (C == 1) {
                xi = __fdiv_rn(1.f, __fadd_rn(1.f, expf(-xs[0])));
            } else {
                float xm = -FLT_MAX;
                for (int c = lane; c < C; c += G) xm = fmaxf(xm, xs[c]);
                xm = grp_max<G>(gmask, xm);
                float Sx = 0.f;
                for (int c = lane; c < C; c += G) Sx += expf(xs[c] - xm);
                Sx = grp_sum<G>(gmask, Sx);
                xi = __fdiv_rn(1.f, Sx);
            }
        }
        const bool exit_ok = have_xi && (xi >= pJ);

        // Token-similarity exit prediction (Eq. 36): nearest centroid by cosine
        // (score h.c_j / |c_j|, ties to the lower index); layers >= L_hat are
        // predicted not to run and leave the look-ahead.
        int Lhat = p.N;
        if (p.n_cent > 0) {
            float bsc = -kInf;
            int bj = 0x7fffffff;
            for (int j0 = lane; j0 < p.n_cent; j0 += kMS * G) {
                const int nv = min(kMS, (p.n_cent - j0 + G - 1) / G);
                float acc[kMS];
                multi_sum(zrow, kstride, p.ksplit, E + C + j0, G, nv, acc);
#pragma unroll
                for (int u = 0; u < kMS; ++u) {
                    if (u >= nv) continue;
                    const int j = j0 + u * G;
                    const float cn = p.cnorm[j];
                    const float sc = cn > 0.f ? __fdiv_rn(acc[u], cn) : -kInf;
                    if (sc > bsc || (sc == bsc && j < bj)) { bsc = sc; bj = j; }
                }
            }
            grp_argmax<G>(gmask, bsc, bj);
            Lhat = p.lhat_tab[bj];
        }
        if (lane == 0 && p.lhat_out) p.lhat_out[t] = (int16_t)Lhat;

        // Transmission necessity (Eq. 35) over the budget-feasible candidates (Eq. 34).
        float Gamma = 0.f;
        for (int j = 0; j < K; ++j) {
            const int c0 = coff_l[topk[j]], c1 = coff_l[topk[j] + 1];
            float gmin = kInf;
            for (int c = c0 + lane; c < c1; c += G) {
                const float Q = p.tab.cand_Q[c];
                if (__fadd_rn(Dhat, Q) <= Dbar) {
                    const int m = p.tab.cand_m[c];
                    gmin = fminf(gmin, (m != s) ? p.tab.trans[s * M + m] : 0.f);
                }
            }
            Gamma = __fadd_rn(Gamma, grp_min<G>(gmask, gmin));
        }
        const float Lambda = __fmul_rn(p.tab.lambda[l], I);
        const bool skip_ok = (Gamma > 0.f) && (I <= p.tab.theta[l]) && (__fadd_rn(Dhat, Lambda) <= Dbar);

        // Look-ahead Phi^{(H-1)}_l over all (m, k), bottom-up (Eq. 39).  Phi
        // depends on the token only through Dbar and the tests Q <= R and
        // eps <= R, so every R between two consecutive thresholds of the window
        // gives the same table: with the layer's Dbar the token reads the table
        // of its interval, computed once with the same operation order.
        const float R = __fsub_rn(Dbar, Dhat);
        const int top = max(0, min(min(p.H - 1, p.N - 1 - l), Lhat - 1 - l));
        bool have_phi = false;
        const float* phiP = bufPhi;
        const bool use_shared = p.phi_tabs != nullptr && top >= p.dmin && top > 0 && Dbar == *p.dbar_shared;
        if (use_shared) {
            int lo = 0, hi = p.n_thr;       // interval = number of thresholds <= R
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (p.thr[mid] <= R) lo = mid + 1; else hi = mid;
            }
            phiP = p.phi_tabs + ((size_t)(top - p.dmin) * (p.n_thr + 1) + lo) * ME;
            have_phi = true;
        }
        for (int jj = use_shared ? 0 : top; jj >= 1; --jj) {
            const int lp = l + jj;
            const float eps = p.tab.eps[lp];
            const int* coff = p.tab.cand_off + lp * (E + 1);
            const int cb = coff[0];
            const int nc = coff[E] - cb;
            // (1) per-candidate terms
            for (int c = lane; c < nc; c += G) {
                const float Q = p.tab.cand_Q[cb + c];
                const int mm = p.tab.cand_m[cb + c];
                cok[c] = (Q <= R) ? 1 : 0;
                cqt[c] = (Q > 0.f) ? __fmul_rn(p.omega_D, __fdiv_rn(Q, Dbar)) : -1.f;
                cph[c] = have_phi ? bufPhi[mm * E + p.tab.cand_k[cb + c]] : 0.f;
                cmv[c] = (uint8_t)mm;
            }
            __syncwarp(gmask);
            // (2) V(m, k') = best next action from m for target k'
            const float* ct = p.tab.ctab + (size_t)lp * M * M;
            const float skip_cost = __fmul_rn(p.omega_D, __fdiv_rn(eps, Dbar));
            const bool skip_budget = eps <= R;
            for (int idx = lane; idx < ME; idx += G) {
                const int m = idx / E, kp = idx - (idx / E) * E;
                const int s0 = coff[kp] - cb, s1 = coff[kp + 1] - cb;
                const float* ctm = ct + m * M;
                float best = kInf;
                bool local = false;
                for (int c = s0; c < s1; ++c) {
                    if (!cok[c]) continue;
                    const int mm = cmv[c];
                    float v = ctm[mm];
                    const float q = cqt[c];
                    if (q >= 0.f) v = __fadd_rn(v, q);
                    if (have_phi) v = __fadd_rn(v, cph[c]);
                    best = fminf(best, v);
                    local |= (mm == m);
                }
                if (!local && skip_budget) {
                    float v = skip_cost;
                    if (have_phi) v = __fadd_rn(v, bufPhi[m * E + kp]);
                    best = fminf(best, v);
                }
                bufV[idx] = best;
            }
            __syncwarp(gmask);
            // (3) Phi_{l'-1}(m, k)
            const float* Pl = p.tab.P + (size_t)(lp - 1) * E * E;
            for (int idx = lane; idx < ME; idx += G) {
                const int m = idx / E, k = idx - (idx / E) * E;
                const float* Prow = Pl + k * E;
                const float* Vrow = bufV + m * E;
                float acc = 0.f;
                for (int kp = 0; kp < E; ++kp) acc = __fadd_rn(acc, __fmul_rn(__ldg(Prow + kp), Vrow[kp]));
                bufPhi[idx] = acc;
            }
            __syncwarp(gmask);
            have_phi = true;
        }

        // Execute plan: slot 0 by f + Phi, later slots by f (Eq. 40), budget by Eq. (34).
        const float* ct_s = ct_l + s * M;
        int esel[kMaxK], msel[kMaxK];
        float Drun = Dhat, tot = 0.f;
        for (int j = 0; j < K; ++j) {
            const int c0 = coff_l[topk[j]], c1 = coff_l[topk[j] + 1];
            float bv = kInf;
            int bi = 0x7fffffff;
            for (int c = c0 + lane; c < c1; c += G) {
                const float Q = p.tab.cand_Q[c];
                const int m = p.tab.cand_m[c];
                const float ct = ct_s[m];
                // the cost-to-go is read before the budget tests decide whether it is used
                const float ph = (j == 0 && have_phi) ? phiP[m * E + p.tab.cand_k[c]] : 0.f;
                if (!(__fadd_rn(Dhat, Q) <= Dbar)) continue;
                if (!(__fadd_rn(Drun, Q) <= Dbar)) continue;
                float f = ct;
                if (Q > 0.f) f = __fadd_rn(f, __fmul_rn(p.omega_D, __fdiv_rn(Q, Dbar)));
                float v = f;
                if (j == 0) v = __fadd_rn(f, ph);
                if (v < bv) { bv = v; bi = c; }
            }
            grp_argmin<G>(gmask, bv, bi);
            esel[j] = p.tab.cand_k[bi];
            msel[j] = p.tab.cand_m[bi];
            Drun = __fadd_rn(Drun, p.tab.cand_Q[bi]);
            tot = (j == 0) ? bv : __fadd_rn(tot, bv);
        }
        const float tot_exec = tot;
        float tot_skip = kInf;
        if (skip_ok)
            tot_skip = __fadd_rn(__fmul_rn(p.omega_D, __fdiv_rn(Lambda, Dbar)),
                                 have_phi ? phiP[s * E + topk[0]] : 0.f);
        int action = 0;
        float best = tot_exec;
        if (skip_ok && tot_skip < tot_exec) { action = 1; best = tot_skip; }
        if (exit_ok && best > 0.f) action = 2;

        // Outputs and state update (Eq. 41, 42, exit).
        if (lane < K) {
            p.topk_idx[t * K + lane] = topk[lane];
            p.topk_g[t * K + lane] = g[lane];
            p.exp_sel[t * K + lane] = action == 0 ? (uint8_t)esel[lane] : 0xFF;
            p.srv_sel[t * K + lane] = action == 0 ? (uint8_t)msel[lane] : 0xFF;
        }
        if (lane == 0 && p.calib) {
            // Calibration counts of the offline stage (Eq. 26-28, 38).
            atomicAdd(&p.c_alive[l], 1ull);
            atomicAdd(&p.c_resid[l * M + s], 1ull);
            for (int j = 0; j < K; ++j) {
                atomicAdd(&p.c_act[l * E + topk[j]], 1ull);
                if (I > p.tab.theta[l]) atomicAdd(&p.c_above[l * E + topk[j]], 1ull);
            }
            const int prev = p.prev_target[t];
            if (l > 0 && prev >= 0) atomicAdd(&p.c_trans[((size_t)(l - 1) * E + prev) * E + topk[0]], 1ull);
            p.prev_target[t] = (int16_t)topk[0];
        }
        if (lane == 0) {
            p.action[t] = (uint8_t)action;
            p.I_out[t] = I;
            p.xi_out[t] = xi;
            if (xi >= 0.f) p.xi_last[t] = xi;
            float Dnew = Dhat;
            if (action == 0) {
                p.s[t] = (uint8_t)msel[0];
                Dnew = Drun;
                p.Dhat[t] = Dnew;
                p.last_exec[t] = 1;
                float dl = 0.f;
#pragma unroll
                for (int j = 0; j < kMaxK; ++j) {
                    if (j >= K) break;
                    const bool remote = msel[j] != s;
                    const bool sub = esel[j] != topk[j];
                    if (remote) { if (sub) ++wc.rs; else ++wc.re; ++wc.hops; }
                    else { if (sub) ++wc.ls; else ++wc.le; }
                    const float tr = remote ? p.tab.trans[s * M + msel[j]] : 0.f;
                    dl += tr + p.tab.comp[l * M + msel[j]];
                }
                wc.delay += dl;
                ++wc.exec_tokens;
            } else if (action == 1) {
                Dnew = __fadd_rn(Dhat, Lambda);
                p.Dhat[t] = Dnew;
                p.last_exec[t] = 0;
                ++wc.skipped;
            } else {
                p.alive[t] = 0;
                p.exit_layer[t] = (int16_t)l;
                ++wc.exited;
            }
            ++wc.layer_tokens;
            if (use_shared) ++wc.shared_phi;
            if (Dbar > 0.f && Dbar < FLT_MAX) wc.max_ratio = fmaxf(wc.max_ratio, Dnew / Dbar);
        }
        __syncwarp(gmask);
    }
    if (lane == 0) {
        atomicAdd(&blk_cnt[0], wc.layer_tokens);
        atomicAdd(&blk_cnt[1], wc.exec_tokens);
        atomicAdd(&blk_cnt[2], wc.skipped);
        atomicAdd(&blk_cnt[3], wc.exited);
        atomicAdd(&blk_cnt[4], wc.le);
        atomicAdd(&blk_cnt[5], wc.ls);
        atomicAdd(&blk_cnt[6], wc.re);
        atomicAdd(&blk_cnt[7], wc.rs);
        atomicAdd(&blk_cnt[8], wc.hops);
        atomicAdd(&blk_cnt[9], wc.shared_phi);
        atomicAdd(&blk_delay, (double)wc.delay);
        atomicMax(&blk_ratio, __float_as_uint(fmaxf(wc.max_ratio, 0.f)));
    }
    __syncthreads();
    if (threadIdx.x == 0 && blk_cnt[0]) {
        DevCounters* c = p.ctr + (blockIdx.x % kCtrCopies);
        atomicAdd(&c->layer_tokens, blk_cnt[0]);
        atomicAdd(&c->exec_tokens, blk_cnt[1]);
        atomicAdd(&c->skipped, blk_cnt[2]);
        atomicAdd(&c->exited, blk_cnt[3]);
        atomicAdd(&c->pairs_local_exact, blk_cnt[4]);
        atomicAdd(&c->pairs_local_sub, blk_cnt[5]);
        atomicAdd(&c->pairs_remote_exact, blk_cnt[6]);
        atomicAdd(&c->pairs_remote_sub, blk_cnt[7]);
        atomicAdd(&c->remote_hops, blk_cnt[8]);
        atomicAdd(&c->lookahead_shared, blk_cnt[9]);
        atomicAdd(&c->delay_ms, blk_delay);
        atomicMax(&c->max_budget_ratio_bits, blk_ratio);
    }
    pdl_trigger();   // the next kernel may be scheduled once every block got here or exited
}

// One look-ahead table for Dbar = Dbar[0]: layer l, interval iv (R =
// thr[iv - 1], or -inf for iv = 0), depth top (levels l + top .. l + 1), each
// entry by one thread with the same operation order as the per-token path
// above, written to out.  A block has a thread per entry (up to 1024): each
// entry is a chain of dependent loads and roundings, so a table is
// latency-bound.  Called by whole blocks.
__device__ __forceinline__ void lookahead_table(const DecideParams& p, int l, const float* thr, int iv, int top,
                                                float* out) {
    extern __shared__ float smem[];
    const int E = p.E, M = p.M;
    const int ME = M * E;
    const int MC = p.tab.max_layer_cand;
    float* bufV = smem;
    float* bufPhi = bufV + ME;
    float* cqt = bufPhi + ME;
    float* cph = cqt + MC;
    uint8_t* cok = reinterpret_cast<uint8_t*>(cph + MC);
    uint8_t* cmv = cok + ((MC + 3) & ~3);
    const float Dbar = p.Dbar[0];
    const float R = iv == 0 ? -kInf : thr[iv - 1];
    bool have_phi = false;
    for (int jj = top; jj >= 1; --jj) {
        const int lp = l + jj;
        const float eps = p.tab.eps[lp];
        const int* coff = p.tab.cand_off + lp * (E + 1);
        const int cb = coff[0];
        const int nc = coff[E] - cb;
        for (int c = threadIdx.x; c < nc; c += blockDim.x) {
            const float Q = p.tab.cand_Q[cb + c];
            const int mm = p.tab.cand_m[cb + c];
            cok[c] = (Q <= R) ? 1 : 0;
            cqt[c] = (Q > 0.f) ? __fmul_rn(p.omega_D, __fdiv_rn(Q, Dbar)) : -1.f;
            cph[c] = have_phi ? bufPhi[mm * E + p.tab.cand_k[cb + c]] : 0.f;
            cmv[c] = (uint8_t)mm;
        }
        __syncthreads();
        const float* ct = p.tab.ctab + (size_t)lp * M * M;
        const float skip_cost = __fmul_rn(p.omega_D, __fdiv_rn(eps, Dbar));
        const bool skip_budget = eps <= R;
        for (int idx = threadIdx.x; idx < ME; idx += blockDim.x) {
            const int m = idx / E, kp = idx - (idx / E) * E;
            const int s0 = coff[kp] - cb, s1 = coff[kp + 1] - cb;
            const float* ctm = ct + m * M;
            float best = kInf;
            bool local = false;
            for (int c = s0; c < s1; ++c) {
                if (!cok[c]) continue;
                const int mm = cmv[c];
                float v = ctm[mm];
                const float q = cqt[c];
                if (q >= 0.f) v = __fadd_rn(v, q);
                if (have_phi) v = __fadd_rn(v, cph[c]);
                best = fminf(best, v);
                local |= (mm == m);
            }
            if (!local && skip_budget) {
                float v = skip_cost;
                if (have_phi) v = __fadd_rn(v, bufPhi[m * E + kp]);
                best = fminf(best, v);
            }
            bufV[idx] = best;
        }
        __syncthreads();
        const float* Pl = p.tab.P + (size_t)(lp - 1) * E * E;
        for (int idx = threadIdx.x; idx < ME; idx += blockDim.x) {
            const int m = idx / E, k = idx - (idx / E) * E;
            const float* Prow = Pl + k * E;
            const float* Vrow = bufV + m * E;
            float acc = 0.f;
            for (int kp = 0; kp < E; ++kp) acc = __fadd_rn(acc, __fmul_rn(__ldg(Prow + kp), Vrow[kp]));
            bufPhi[idx] = acc;
        }
        __syncthreads();
        have_phi = true;
    }
    for (int idx = threadIdx.x; idx < ME; idx += blockDim.x) out[idx] = have_phi ? bufPhi[idx] : 0.f;
    if (threadIdx.x == 0 && iv == 0) *p.dbar_shared_out = Dbar;
}

// The tables of one layer: block (i, y) computes interval i at depth dmin + y.
__global__ void __launch_bounds__(1024) lookahead_shared_kernel(const DecideParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    const int iv = blockIdx.x;
    lookahead_table(p, p.layer, p.thr, iv, p.dmin + (int)blockIdx.y,
                    p.phi_tabs_out + ((size_t)blockIdx.y * (p.n_thr + 1) + iv) * p.M * p.E);
    pdl_trigger();   // the next kernel may be scheduled once every block got here or exited
}

// The tables of every layer at once (they depend only on the tables, the
// budget Dbar[0] and the cost weights): block (i, y, l) computes interval i at
// depth dmin_l + y of layer l.
__global__ void __launch_bounds__(1024) lookahead_all_kernel(const DecideParams p, const LaLayer* __restrict__ lay) {
    const int l = blockIdx.z;
    const LaLayer L = lay[l];
    const int iv = blockIdx.x, y = blockIdx.y;
    if (L.n_depth <= 0 || iv > L.n_thr || y >= L.n_depth) return;
    const int top_full = min(p.H - 1, p.N - 1 - l);
    lookahead_table(p, l, p.thr + L.thr_off, iv, top_full - L.n_depth + 1 + y,
                    p.phi_tabs_out + L.tab_off + ((size_t)y * (L.n_thr + 1) + iv) * p.M * p.E);
}

}  // namespace

cudaError_t launch_lookahead_shared(const DecideParams& p, int n_depth, cudaStream_t st) {
    if (p.T <= 0 || n_depth <= 0) return cudaSuccess;
    const size_t MC = (size_t)p.tab.max_layer_cand;
    // At most 2 * 1024 + 2 * 1024 floats plus 2 KB of flags (M * E <= 1024): under 48 KB.
    const size_t smem = (2 * (size_t)p.M * p.E + 2 * MC) * sizeof(float) + ((MC + 3) / 4) * 2 * sizeof(float);
    // A plain launch: measured with programmatic serialisation this kernel cost
    // 60 us per layer more on the Qwen-shaped layer (E = 60) and saved nothing
    // elsewhere.
    const int ME = p.M * p.E;
    const int threads = std::min(1024, std::max(256, (ME + 31) / 32 * 32));
    lookahead_shared_kernel<<<dim3(p.n_thr + 1, n_depth), threads, smem, st>>>(p);
    return cudaGetLastError();
}

cudaError_t launch_lookahead_all(const DecideParams& p, const LaLayer* layers, int n_layers, int max_thr,
                                 int max_depth, cudaStream_t st) {
    if (p.T <= 0 || n_layers <= 0 || max_depth <= 0) return cudaSuccess;
    const size_t MC = (size_t)p.tab.max_layer_cand;
    const size_t smem = (2 * (size_t)p.M * p.E + 2 * MC) * sizeof(float) + ((MC + 3) / 4) * 2 * sizeof(float);
    const int ME = p.M * p.E;
    const int threads = std::min(1024, std::max(256, (ME + 31) / 32 * 32));
    lookahead_all_kernel<<<dim3(max_thr + 1, max_depth, n_layers), threads, smem, st>>>(p, layers);
    return cudaGetLastError();
}

// Lanes per token: the smallest group that holds one expert per lane.
int decide_group(int E) { return E <= 8 ? 8 : E <= 16 ? 16 : 32; }

size_t decide_la_floats(int E, int M, int max_layer_cand) {
    const size_t MC = (size_t)max_layer_cand;
    return (size_t)2 * M * E + 2 * MC + ((MC + 3) / 4) * 2;
}

size_t decide_smem_for(int E, int C, int M, int max_layer_cand, int G, bool la_global = false) {
    const size_t per_group = (size_t)(2 * E + C) + (la_global ? 0 : decide_la_floats(E, M, max_layer_cand));
    return per_group * sizeof(float) * kWarps * (32 / G);
}

// Blocks of the decision kernel when the look-ahead scratch is global: at most
// this many per SM (the register-limited occupancy is seven).
constexpr int kDecideLaBlocksPerSm = 8;

// Lanes per token for large batches: a lane per expert up to 16 experts; above
// that 16 lanes (several experts per lane, two tokens per warp), which keeps
// more tokens in flight (Qwen-shaped, E = 60: decide 1.54 -> 1.32 ms per
// forward against a full warp per token), unless the per-token look-ahead
// scratch of eight groups per block does not fit in shared memory.
int decide_group_for(int E, int C, int M, int max_layer_cand) {
    const int g = decide_group(E);
    if (g == 32 && decide_smem_for(E, C, M, max_layer_cand, 16) <= 200 * 1024) return 16;
    return g;
}

size_t decide_la_scratch_floats(int E, int M, int max_layer_cand, int num_sms) {
    return (size_t)num_sms * kDecideLaBlocksPerSm * kWarps * (32 / decide_group(E) > 2 ? 32 / decide_group(E) : 2) *
           decide_la_floats(E, M, max_layer_cand);
}

size_t decide_smem_bytes(int E, int C, int M, int max_layer_cand) {
    return decide_smem_for(E, C, M, max_layer_cand, decide_group(E));
}

cudaError_t launch_decide(const DecideParams& p, int num_sms, cudaStream_t st) {
    if (p.T <= 0) return cudaSuccess;
    // Groups smaller than a warp pay off when the tokens outnumber the resident
    // warps (seven 4-warp blocks per SM); up to that many tokens keep a full
    // warp per token for the shortest per-token latency (its look-ahead loops
    // run over M*E entries): the Switch-shaped layer of 4096 tokens 1.008 ->
    // 0.980 ms per forward against lane groups of 8.
    const int G = p.T > num_sms * 7 * kWarps ? decide_group_for(p.E, p.C, p.M, p.tab.max_layer_cand) : 32;
    const bool la_global = p.la_scratch != nullptr;
    const size_t smem = decide_smem_for(p.E, p.C, p.M, p.tab.max_layer_cand, G, la_global);
    static PerDevice attr;
    const cudaError_t ea = (cudaError_t)attr.get([] {
        cudaError_t e = cudaFuncSetAttribute(decide_kernel<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(decide_kernel<16>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        if (e == cudaSuccess)
            e = cudaFuncSetAttribute(decide_kernel<32>, cudaFuncAttributeMaxDynamicSharedMemorySize, 200 * 1024);
        return (int)e;
    }, true);
    if (ea != cudaSuccess) return ea;
    if (smem > 200 * 1024) return cudaErrorInvalidValue;
    const int per_block = kWarps * (32 / G);
    int blocks = (p.T + per_block - 1) / per_block;
    const int cap = la_global ? num_sms * kDecideLaBlocksPerSm : num_sms * 16;   // global slots exist for cap blocks
    blocks = blocks < cap ? blocks : cap;
    cudaError_t e;
    if (G == 8) e = launch_pdl(decide_kernel<8>, dim3(blocks), dim3(kWarps * 32), smem, st, p);
    else if (G == 16) e = launch_pdl(decide_kernel<16>, dim3(blocks), dim3(kWarps * 32), smem, st, p);
    else e = launch_pdl(decide_kernel<32>, dim3(blocks), dim3(kWarps * 32), smem, st, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
