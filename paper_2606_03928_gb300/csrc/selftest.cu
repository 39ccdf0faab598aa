// Self-test of the failure detection: a kernel whose bounded wait cannot complete.
//
// Every wait of the library's kernels (on an mbarrier phase) gives up after kWaitLimitCycles, records its
// site in the device error word and lets the kernel finish, so a stalled pipeline surfaces as an error
// status on the host instead of a hung GPU.  This kernel exercises that path on purpose without a fault:
// one thread waits on a freshly initialised mbarrier that nothing ever arrives at, the wait runs out (about
// two seconds at 2 GHz), the site kSelfTestSite is recorded, and the kernel returns.
#include "ptx.cuh"

namespace vase {

namespace {

constexpr uint32_t kSelfTestSite = 127;

__global__ void wait_timeout_kernel(uint32_t* err) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    mbar_init(&bar, 1);
    fence_mbar_init();
    mbar_wait(&bar, 0, err, kSelfTestSite);  // no arrival ever completes phase 0
}

}  // namespace

cudaError_t launch_wait_timeout_probe(uint32_t* err, cudaStream_t s) {
    wait_timeout_kernel<<<1, 32, 0, s>>>(err);
    return cudaGetLastError();
}

}  // namespace vase
