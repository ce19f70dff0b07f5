// selftest.cu -- exercises the failure path of the library's bounded waits.
//
// Every mbarrier wait in the grouped GEMM gives up after a time limit, sets the
// device status word to VMOE_ERR_DEVICE_TIMEOUT and lets the kernel return, so a
// stalled pipeline surfaces as an error the host can read instead of a hung GPU.
// This kernel waits on an mbarrier that nothing ever arrives on, with a short
// limit, through the same wait routine, so that path can be tested on a GPU
// without faulting or hanging it.
#include "gemm_tc.cuh"

namespace vmoe {
namespace {

__global__ void bounded_wait_selftest_kernel(unsigned long long limit_ns, int *status) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        tc::mbar_init(tc::smem_u32(&bar), 1);
        abort_flag = 0;
        tc::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0)  // phase 0 never completes: the wait must run out
        tc::wait_phase(tc::smem_u32(&bar), 0, &abort_flag, status, limit_ns);
}

}  // namespace
}  // namespace vmoe

extern "C" int vmoe_selftest_bounded_wait(long long limit_ns, void *cuda_stream) {
    if (limit_ns <= 0 || limit_ns > 1000000000LL) return VMOE_ERR_INVALID;
    int *status = vmoe::device_status_word();
    if (!status) return VMOE_ERR_CUDA;
    vmoe::bounded_wait_selftest_kernel<<<1, 32, 0, (cudaStream_t)cuda_stream>>>(
        (unsigned long long)limit_ns, status);
    return vmoe::launch_result();
}
