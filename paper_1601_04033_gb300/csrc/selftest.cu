// Self-test of the failure path of the dense pass's copy pipeline: one block
// whose pipeline barrier never completes (it expects one arrival and none
// comes), waited on with the pass's own bounded waits -- by one thread (the
// producer's form, wait_one) and by a whole warp (the consumers' form,
// wait_warp), at the same time.  Each wait gives up after about a second and
// raises kErrWaitTimeout in the error word; the kernel then returns.  No copy
// is in flight, nothing traps, and the context stays usable.

#include "kernels.cuh"
#include "wait.cuh"

namespace fasgd {
namespace {

__global__ void __launch_bounds__(64) wait_expiry_kernel(int32_t* err) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (threadIdx.x == 0) wait_one(&bar, 0, err);
    if (threadIdx.x >= 32) wait_warp(&bar, 0, err);
}

}  // namespace

cudaError_t launch_wait_expiry(int32_t* err, cudaStream_t stream) {
    wait_expiry_kernel<<<1, 64, 0, stream>>>(err);
    return cudaGetLastError();
}

}  // namespace fasgd
