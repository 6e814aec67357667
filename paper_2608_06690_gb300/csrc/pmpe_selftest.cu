// pmpe_selftest_wait_timeout: exercises the bounded mbarrier wait that every
// pipeline stage of the layer's tensor-core kernels uses, on a barrier that
// nothing ever arrives on, so that a test can check that an expired wait
// records PMPE_STATUS_PIPELINE_TIMEOUT and returns instead of hanging, and
// that the CUDA context stays usable afterwards.
#include "pmpe_internal.cuh"
#include "tc_ptx.cuh"

namespace pmpe {
namespace {

__global__ void wait_timeout_kernel(uint32_t *status, unsigned long long limit_ns)
{
    __shared__ __align__(8) uint64_t bar;
    __shared__ volatile int abort_flag;
    if (threadIdx.x != 0) return;
    abort_flag = 0;
    const uint32_t b = smem_u32(&bar);
    mbar_init(b, 1);  // expects one arrival, which never comes
    asm volatile("fence.mbarrier_init.release.cluster;\n" ::: "memory");
    mbar_wait_for(b, 0, &abort_flag, status, limit_ns);
}

}  // namespace
}  // namespace pmpe

extern "C" int pmpe_selftest_wait_timeout(uint32_t *status, int limit_us, void *stream)
{
    if (!status || limit_us < 1 || limit_us > 1000000) return PMPE_ERR_INVALID_ARG;
    pmpe::wait_timeout_kernel<<<1, 32, 0, (cudaStream_t)stream>>>(status, 1000ull * (unsigned long long)limit_us);
    return cudaGetLastError() == cudaSuccess ? PMPE_OK : PMPE_ERR_CUDA;
}
