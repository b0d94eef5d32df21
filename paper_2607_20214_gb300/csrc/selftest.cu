// Self-test of the in-band failure path (elsaa_selftest_wait_timeout).
#include "device_common.cuh"
#include "tc_common.cuh"

namespace elsaa {

namespace {

// One thread waits, with the kernels' own bounded-wait routine, on an
// mbarrier that nothing arrives on: after limit_ns the wait gives up, the
// status word records kDevWaitTimeout at site 0x7e57 and the kernel
// returns. No fault, no hang: the context stays usable.
__global__ void k_selftest_wait(DeviceStatus *status,
                                unsigned long long limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    tc::mbar_init(&bar, 1);
    tc::fence_mbar_init();
    tc::mbar_wait_limit(&bar, 0, status, 0x7e57, limit_ns);
}

}  // namespace

cudaError_t launch_selftest_wait(DeviceStatus *status, int limit_ms,
                                 cudaStream_t st) {
    k_selftest_wait<<<1, 32, 0, st>>>(
        status, (unsigned long long)limit_ms * 1000000ull);
    return cudaGetLastError();
}

}  // namespace elsaa
