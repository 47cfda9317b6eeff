// selftest.cu -- a check of the failure-detection path.  One kernel waits on
// an mbarrier that no thread arrives on, through the same bounded wait the
// scan kernels use for their pipeline barriers.  The wait gives up after
// kWaitLimitNs and the kernel records NEST_ERR_TIMEOUT in the datastore's
// status word, as a scan kernel does when a stage never arrives; nothing
// faults or hangs, and the context stays usable.
#include "internal.h"
#include "ptx.cuh"

namespace nest {
namespace {

__global__ void bounded_wait_selftest_kernel(int* status, int64_t* waited_ns)
{
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);  // phase 0 completes on one arrival; none comes
        mbar_init_fence();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        const uint64_t t0 = global_timer_ns();
        if (!mbar_wait_bounded(&bar, 0)) record_status(status, NEST_ERR_TIMEOUT);
        *waited_ns = (int64_t)(global_timer_ns() - t0);
    }
}

}  // namespace

cudaError_t launch_wait_selftest(int* status, int64_t* waited_ns, cudaStream_t stream)
{
    bounded_wait_selftest_kernel<<<1, 32, 0, stream>>>(status, waited_ns);
    return cudaGetLastError();
}

}  // namespace nest
