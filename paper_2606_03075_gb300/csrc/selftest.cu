// Self-test of the failure detection: one bounded wait that runs out.
//
// Every kernel of the library waits on its mbarriers with tc::mbar_wait, which
// gives up after a fixed number of SM cycles and lets the kernel set
// TGVKV_STATUS_TIMEOUT instead of hanging.  This kernel makes exactly that wait
// on a barrier that no thread arrives at, so that a test can check, on a GPU,
// that the wait ends, the status word records it and the context stays usable.
#include "common.cuh"
#include "launch.h"
#include "tc05.cuh"

namespace tgvkv {
namespace {

__global__ void wait_timeout_kernel(uint32_t* __restrict__ status) {
    __shared__ uint64_t bar;
    __shared__ int never;
    if (threadIdx.x == 0) {
        never = 0;
        tc::mbar_init(&bar, 1);
        tc::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // phase 0 of `bar` never completes: nothing arrives
        if (!tc::mbar_wait(&bar, 0, &never)) raise_status(status, TGVKV_STATUS_TIMEOUT);
    }
}

}  // namespace

cudaError_t launch_wait_timeout(uint32_t* status, cudaStream_t stream) {
    wait_timeout_kernel<<<1, 32, 0, stream>>>(status);
    return cudaGetLastError();
}

}  // namespace tgvkv
