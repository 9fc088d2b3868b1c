// selftest.cu -- logo_selftest_wait_expiry: exercises the library's bounded
// waits without a fault.  One warp waits on an mbarrier that nothing will ever
// arrive at, through the same wait every pipelined kernel uses; after the
// given budget the wait gives up, records LOGO_ERR_TIMEOUT in the device
// status word, and the block returns normally.  The context stays usable.
#include <cuda_runtime.h>

#include <cstdint>

#include "host_common.h"
#include "sm100.cuh"

namespace logo {
namespace {

__global__ void __launch_bounds__(32) wait_expiry_kernel(uint64_t budget_ns)
{
    __shared__ __align__(8) uint64_t bar;
    __shared__ volatile int abort_flag;
    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar), 1);  // one arrival expected, none will come
        fence_mbar_init();
    }
    __syncwarp();
    mbar_wait(smem_u32(&bar), 0, &abort_flag, budget_ns);  // phase 0 never completes
}

}  // namespace

int selftest_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" int logo_selftest_wait_expiry(uint64_t budget_ns, void* stream)
{
    if (budget_ns == 0 || budget_ns > kWaitBudgetNs) return LOGO_ERR_INVALID_ARG;
    wait_expiry_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(budget_ns);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
