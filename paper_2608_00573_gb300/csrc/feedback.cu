// Runtime feedback between forwards (the periodic update of Algorithm 2, Sec. V-D/V-F).
//
// Eq. (37): for every user (a block of user_size consecutive tokens) with exits
// in the observation window, p_J <- clamp(p_J + eta * (mean exit confidence -
// p_J), p_min, 1).  The per-user utilisation sum(Dhat) / sum(Dbar) feeds the
// dual-weight update of Eq. (43), finished on the host.  One thread per user
// sums its tokens in order, and one thread sums the users in order, so the
// results do not depend on scheduling.
#include "internal.cuh"

namespace tmoe {

namespace {

__global__ void __launch_bounds__(128) feedback_users_kernel(const FeedbackParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    const int u = blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= p.users) return;
    const int t0 = u * p.user_size;
    const int t1 = min(p.T, t0 + p.user_size);
    double xs = 0.0, dh = 0.0, db = 0.0;
    int n = 0;
    for (int t = t0; t < t1; ++t) {
        if (!p.alive[t] && p.exit_layer[t] < p.N) {
            xs += (double)p.xi_last[t];
            ++n;
        }
        dh += (double)p.Dhat[t];
        db += (double)p.Dbar[t];
    }
    if (n > 0) {
        const float xbar = (float)(xs / n);
        for (int t = t0; t < t1; ++t) {
            const float pj = p.pJ[t];
            float q = __fadd_rn(pj, __fmul_rn(p.eta, __fsub_rn(xbar, pj)));
            q = fminf(fmaxf(q, p.p_min), 1.f);
            p.pJ[t] = q;
        }
    }
    p.util[u] = (db > 0.0) ? dh / db : 0.0;
    p.updated[u] = n > 0 ? 1 : 0;
}

__global__ void feedback_reduce_kernel(const FeedbackParams p) {
    pdl_wait();      // results of the preceding kernel in the stream
    pdl_trigger();   // single-wave grid: let the next kernel be scheduled now
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    double s = 0.0;
    int n = 0;
    for (int u = 0; u < p.users; ++u) {
        s += p.util[u];
        n += p.updated[u];
    }
    p.result[0] = p.users > 0 ? s / p.users : 0.0;
    p.result[1] = (double)n;
}

}  // namespace

cudaError_t launch_feedback(const FeedbackParams& p, cudaStream_t st) {
    cudaError_t e = cudaSuccess;
    if (p.users > 0) e = launch_pdl(feedback_users_kernel, dim3((p.users + 127) / 128), dim3(128), 0, st, p);
    if (e == cudaSuccess) e = launch_pdl(feedback_reduce_kernel, dim3(1), dim3(32), 0, st, p);
    if (e != cudaSuccess) return e;
    return cudaGetLastError();
}

}  // namespace tmoe
