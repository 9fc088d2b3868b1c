// budget.cu -- the budget controller of Sec. 3.2 on the device.
//
//   logo_budget_update            Eq. 3 realised ratio F = N / (B*T) from the
//                                 selection's device-side count, and the Eq. 11
//                                 threshold step b_th += gamma * sign(F - rho),
//                                 applied to a device-resident b_th
//   logo_pmask_initial_threshold  the P-mask start value (Sec. 3.2, App. C.1)
//
// With logo_select_device_threshold reading the same b_th, a training step's
// routing loop (select -> attention -> ... -> budget update) runs without any
// host synchronisation.  One thread: the work is a handful of scalar
// operations, launched once per layer per step.
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>

#include "host_common.h"

namespace logo {
namespace {

// F and the sign are evaluated in double from the integer counts; b_th and
// gamma are float32 and the update is one float32 addition (gamma * sign is
// exact), so the trajectory is reproducible bit for bit.
__global__ void budget_update_kernel(const int32_t* __restrict__ n_sel_total, long long n_valid, float rho,
                                     float gamma, float* __restrict__ b_th, float* __restrict__ f_out)
{
    if (threadIdx.x != 0 || blockIdx.x != 0) return;
    const double F = static_cast<double>(*n_sel_total) / static_cast<double>(n_valid);
    const double d = F - static_cast<double>(rho);
    const float sgn = d > 0.0 ? 1.0f : (d < 0.0 ? -1.0f : 0.0f);
    *b_th = __fadd_rn(*b_th, gamma * sgn);
    if (f_out) *f_out = static_cast<float>(F);
}

}  // namespace
}  // namespace logo

using namespace logo;

extern "C" int logo_budget_update(const int32_t* n_sel_total, logo_dims dims, float rho, float gamma, float* b_th,
                                  float* f_out, void* stream)
{
    if (dims.B < 1 || dims.T < 1) return LOGO_ERR_INVALID_ARG;
    if (!n_sel_total || !b_th) return LOGO_ERR_INVALID_ARG;
    if (!(rho >= 0.0f && rho <= 1.0f)) return LOGO_ERR_INVALID_ARG;
    if (!(gamma >= 0.0f) || !std::isfinite(gamma)) return LOGO_ERR_INVALID_ARG;
    const long long n_valid = static_cast<long long>(dims.B) * dims.T;
    budget_update_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(n_sel_total, n_valid, rho, gamma, b_th,
                                                                           f_out);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

extern "C" float logo_pmask_initial_threshold(float gamma, long long pmask_steps)
{
    return static_cast<float>(0.5 - static_cast<double>(gamma) * static_cast<double>(pmask_steps));
}
