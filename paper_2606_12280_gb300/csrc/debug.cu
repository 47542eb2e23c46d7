// debug.cu -- test hook for the failure-detection path of the tcgen05 GEMMs.
//
// One warp waits on an mbarrier that nothing ever arrives on, through the same
// bounded wait (tc::mbar_wait) that every GEMM role uses.  The wait gives up
// after `limit_ns`, records ERR_WAIT_PROBE in the library's device error word
// and the kernel returns normally, so the context stays usable.
#include <cstdint>
#include <cuda_runtime.h>

#include "launch.h"
#include "tc_ptx.cuh"

namespace w8a8 {
namespace {

constexpr unsigned int ERR_WAIT_PROBE = 128u;

__global__ void wait_probe_kernel(unsigned int *err, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    const uint32_t b = tc::smem_addr(&bar);
    if (threadIdx.x == 0) {
        tc::mbar_init(b, 1);
        abort_flag = 0;
        tc::fence_barrier_init();
    }
    __syncthreads();
    const tc::WaitCtx wc{tc::smem_addr(&abort_flag), err, limit_ns};
    if (threadIdx.x == 0) (void)tc::mbar_wait(b, 0, wc, ERR_WAIT_PROBE);
    __syncthreads();
}

}  // namespace

cudaError_t launch_wait_probe(unsigned int *err, uint64_t limit_ns, cudaStream_t st) {
    wait_probe_kernel<<<1, 32, 0, st>>>(err, limit_ns);
    return cudaGetLastError();
}

}  // namespace w8a8
