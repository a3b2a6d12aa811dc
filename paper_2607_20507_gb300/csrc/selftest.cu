// selftest.cu -- the failure-detection self-test (cs_selftest_wait_timeout):
// the bounded mbarrier wait of the attention kernels, run on a barrier that
// nothing arrives at.
#include "cs_device.cuh"
#include "cs_internal.h"

namespace cs {

namespace {
// One thread runs the kernels' bounded wait on a barrier that nothing
// arrives at: after about one second the wait gives up and the thread records
// CS_DEVICE_WAIT_TIMEOUT, as a kernel's role would.
__global__ void wait_selftest_kernel(int* status) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    fence_barrier_init();
    if (!mbar_wait_bounded(&bar, 0)) atomicOr(status, CS_DEVICE_WAIT_TIMEOUT);
}
}  // namespace

cudaError_t launch_wait_selftest(int* status, cudaStream_t stream) {
    wait_selftest_kernel<<<1, 32, 0, stream>>>(status);
    return cudaGetLastError();
}

}  // namespace cs
