// Self-check of the bounded device waits (failure detection without a fault).
//
// Every wait of the library's kernels on an mbarrier has a time limit; when it
// runs out the waiting role raises its CTA's abort flag and writes a code to
// the handle's device error word, the other roles see the flag and return, and
// the kernel ends normally.  This kernel exercises exactly that path: its only
// mbarrier never receives an arrival.

#include "internal.cuh"

namespace tmoe {

__global__ void __launch_bounds__(64) watchdog_selftest_kernel(int* err, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        fence_barrier_init();
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (lane == 0) {
        // Phase 0 of a barrier expecting one arrival that never comes.  Warp 0
        // runs out after limit_ns; warp 1 keeps the kernels' normal limit and
        // returns once warp 0 has raised the abort flag.
        if (warp == 0)
            mbar_wait_bounded(smem_u32(&bar), 0, &abort_flag, err, ERR_TIMEOUT_SELFTEST, limit_ns);
        else
            mbar_wait_bounded(smem_u32(&bar), 0, &abort_flag, err, ERR_TIMEOUT_SELFTEST);
    }
    __syncthreads();
}

cudaError_t launch_watchdog_selftest(int* err, uint64_t limit_ns, cudaStream_t st) {
    watchdog_selftest_kernel<<<1, 64, 0, st>>>(err, limit_ns);
    return cudaGetLastError();
}

}  // namespace tmoe
