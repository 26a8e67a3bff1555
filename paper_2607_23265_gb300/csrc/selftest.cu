// Self-test of the bounded shared-memory barrier wait (the same routine the
// relevance, condensation and projector kernels use for their TMA and
// tensor-core handoffs): a barrier that nothing completes must release the
// waiter after the limit, with the timeout recorded for the host.
#include "wz_internal.cuh"
#include "wz_ptx.cuh"

namespace wz {

__global__ void bounded_wait_selftest_kernel(uint64_t timeout_ns, int *status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x != 0) return;
    ptx::mbar_init(&bar, 1);
    ptx::fence_barrier_init();
    // phase 0 of a fresh barrier completes only after one arrival, which
    // never comes: the wait has to give up on its own
    if (!ptx::mbar_wait(&bar, 0u, timeout_ns)) atomicOr(status, WZ_STATUS_WAIT_TIMEOUT);
}

}  // namespace wz

extern "C" int wz_selftest_bounded_wait(uint64_t timeout_ns, int32_t *device_status, wz_stream_t stream) {
    if (!device_status || timeout_ns == 0 || timeout_ns > 1000000000ull) return WZ_ERR_INVALID_ARG;
    wz::bounded_wait_selftest_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(timeout_ns, device_status);
    return cudaGetLastError() == cudaSuccess ? WZ_OK : WZ_ERR_CUDA;
}
