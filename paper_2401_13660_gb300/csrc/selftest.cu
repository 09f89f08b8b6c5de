// Diagnostic of the library's bounded device-side waits (failure detection).
// Every wait in the kernels goes through mbar_wait_for: when the awaited
// phase does not complete within its limit the kernel records MB_ERR_TIMEOUT
// in the caller's status block and returns, instead of hanging the GPU. This
// kernel makes that path run on purpose: one warp waits on an mbarrier that
// nothing ever arrives on, for a caller-chosen number of SM clocks, then
// records the timeout (detail = clocks waited) and exits with no copies in
// flight, so the context stays usable.
#include "common.cuh"
#include "tma.cuh"

namespace mbscan {
namespace {

__global__ void wait_timeout_kernel(StatusBlock *sb, long long limit) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        fence_mbar_init();
    }
    __syncthreads();
    const long long t0 = clock64();
    const bool ok = mbar_wait_for(&bar, 0, limit);   // phase 0 never completes
    if (!ok && threadIdx.x == 0) report(sb, 4 /* MB_ERR_TIMEOUT */, clock64() - t0);
}

}  // namespace

cudaError_t launch_wait_timeout(StatusBlock *sb, long long limit, cudaStream_t s) {
    wait_timeout_kernel<<<1, 32, 0, s>>>(sb, limit);
    return cudaGetLastError();
}

}  // namespace mbscan
