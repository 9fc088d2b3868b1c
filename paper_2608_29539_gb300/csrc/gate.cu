// gate.cu -- logo_gate_select / logo_gate_bwd: the token gate of Eq. 7,
// p_t = sigmoid(x_t . w_g), computed ahead of the selection it feeds (one
// call instead of a caller GEMV, sigmoid and select), and its backward.
//
// HBM-bound.  The forward reads x once: one warp per token, 16-byte vectors
// of 8 bf16, w_g through the read-only cache, fp32 accumulation, a shuffle
// tree, then the sigmoid.  The backward reads x once more and writes
// dx = dlogit w_g (rank one; optionally added to the caller's dx) and
// dw_g = sum_t dlogit_t x_t with dlogit_t = dp_t p_t (1 - p_t): a thread owns
// fixed 8-wide slices of d_model for all the tokens of its block (two tokens
// per step, so the loads of both are in flight together), and the per-block
// sums are added by a second kernel in a fixed order (colsum.cuh:
// deterministic).
#include <cuda_bf16.h>

#include <cstdint>

#include "colsum.cuh"
#include "host_common.h"
#include "sm100.cuh"

namespace logo {
namespace {

constexpr int kFwdThreads = 256;  // 8 warps, one token per warp at a time
constexpr int kBwdThreads = 256;
constexpr int kMaxModel = 8 * kBwdThreads * 4;  // d_model <= 8192 (4 slices of 8 per thread)

__device__ __forceinline__ void unpack8(const uint4& raw, float (&f)[8])
{
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 v = __bfloat1622float2(h[i]);
        f[2 * i] = v.x;
        f[2 * i + 1] = v.y;
    }
}

__device__ __forceinline__ uint4 pack8(const float (&f)[8])
{
    uint4 raw;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(f[2 * i], f[2 * i + 1]);
    return raw;
}

// x_t . w for two tokens of a warp per pass (t and t + the warp count): one
// load of w serves both, and two f32x2 chains per token keep the FMA
// dependency chain a quarter as long as one scalar accumulator's.
__global__ void __launch_bounds__(kFwdThreads) gate_fwd_kernel(const logo_bf16* __restrict__ x,
                                                               const float* __restrict__ w, int64_t ntok, int dm,
                                                               float* __restrict__ p)
{
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (kFwdThreads / 32);
    const int nv = dm / 8;
    for (int64_t t = static_cast<int64_t>(blockIdx.x) * (kFwdThreads / 32) + (threadIdx.x >> 5); t < ntok;
         t += 2 * nwarps) {
        const int64_t t2 = t + nwarps;
        const bool two = t2 < ntok;
        const uint4* xr = reinterpret_cast<const uint4*>(x + t * dm);
        const uint4* xr2 = reinterpret_cast<const uint4*>(x + (two ? t2 : t) * dm);
        uint64_t a0 = 0ull, a1 = 0ull, b0 = 0ull, b1 = 0ull;
#pragma unroll 4
        for (int v = lane; v < nv; v += 32) {
            const float4* wv = reinterpret_cast<const float4*>(w + v * 8);
            const float4 w0 = __ldg(wv), w1 = __ldg(wv + 1);
            const uint64_t wa = f2_pack(w0.x, w0.y), wb = f2_pack(w0.z, w0.w);
            const uint64_t wc = f2_pack(w1.x, w1.y), wd = f2_pack(w1.z, w1.w);
            float xf[8];
            unpack8(xr[v], xf);
            a0 = f2_fma(f2_pack(xf[0], xf[1]), wa, a0);
            a1 = f2_fma(f2_pack(xf[2], xf[3]), wb, a1);
            a0 = f2_fma(f2_pack(xf[4], xf[5]), wc, a0);
            a1 = f2_fma(f2_pack(xf[6], xf[7]), wd, a1);
            if (two) {
                unpack8(xr2[v], xf);
                b0 = f2_fma(f2_pack(xf[0], xf[1]), wa, b0);
                b1 = f2_fma(f2_pack(xf[2], xf[3]), wb, b1);
                b0 = f2_fma(f2_pack(xf[4], xf[5]), wc, b0);
                b1 = f2_fma(f2_pack(xf[6], xf[7]), wd, b1);
            }
        }
        float u0, u1, u2, u3;
        f2_unpack(f2_add(a0, a1), u0, u1);
        f2_unpack(f2_add(b0, b1), u2, u3);
        float a = u0 + u1, b = u2 + u3;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            a += __shfl_xor_sync(0xffffffffu, a, o);
            b += __shfl_xor_sync(0xffffffffu, b, o);
        }
        if (lane == 0) {
            p[t] = 1.0f / (1.0f + expf(-a));
            if (two) p[t2] = 1.0f / (1.0f + expf(-b));
        }
    }
}

// part (when non-null): [gridDim.x][dm] float32 per-block sums of dw_g.
template <int VPT>
__global__ void __launch_bounds__(kBwdThreads) gate_bwd_kernel(const logo_bf16* __restrict__ x,
                                                               const float* __restrict__ w,
                                                               const float* __restrict__ p,
                                                               const float* __restrict__ dp, int64_t ntok, int dm,
                                                               logo_bf16* __restrict__ dx, int accumulate,
                                                               float* __restrict__ part)
{
    const int nv = dm / 8;
    float wr[VPT][8], acc[VPT][8];
#pragma unroll
    for (int k = 0; k < VPT; ++k) {
        const int v = threadIdx.x + k * kBwdThreads;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            wr[k][i] = v < nv ? w[v * 8 + i] : 0.f;
            acc[k][i] = 0.f;
        }
    }
    const int64_t step = gridDim.x;
    for (int64_t t0 = blockIdx.x; t0 < ntok; t0 += 2 * step) {
        const int64_t t1 = t0 + step;
        const bool has1 = t1 < ntok;
        // dlogit = dp p (1 - p), the derivative of the sigmoid at the token's logit
        const float p0 = p[t0], g0 = dp[t0] * p0 * (1.0f - p0);
        const float p1 = has1 ? p[t1] : 0.f, g1 = has1 ? dp[t1] * p1 * (1.0f - p1) : 0.f;
        uint4 x0[VPT], x1[VPT], d0[VPT], d1[VPT];
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kBwdThreads;
            const bool act = v < nv;
            x0[k] = act ? reinterpret_cast<const uint4*>(x + t0 * dm)[v] : make_uint4(0, 0, 0, 0);
            x1[k] = (act && has1) ? reinterpret_cast<const uint4*>(x + t1 * dm)[v] : make_uint4(0, 0, 0, 0);
            d0[k] = (act && dx && accumulate) ? reinterpret_cast<const uint4*>(dx + t0 * dm)[v] : make_uint4(0, 0, 0, 0);
            d1[k] = (act && has1 && dx && accumulate) ? reinterpret_cast<const uint4*>(dx + t1 * dm)[v]
                                                       : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kBwdThreads;
            if (v >= nv) continue;
            float a[8], b[8];
            unpack8(x0[k], a);
            unpack8(x1[k], b);
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[k][i] = fmaf(g1, b[i], fmaf(g0, a[i], acc[k][i]));
            if (dx) {
                float o0[8], o1[8];
                unpack8(d0[k], o0);
                unpack8(d1[k], o1);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    o0[i] = fmaf(g0, wr[k][i], o0[i]);
                    o1[i] = fmaf(g1, wr[k][i], o1[i]);
                }
                reinterpret_cast<uint4*>(dx + t0 * dm)[v] = pack8(o0);
                if (has1) reinterpret_cast<uint4*>(dx + t1 * dm)[v] = pack8(o1);
            }
        }
    }
    if (part) {
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kBwdThreads;
            if (v < nv) {
#pragma unroll
                for (int i = 0; i < 8; ++i) part[static_cast<int64_t>(blockIdx.x) * dm + v * 8 + i] = acc[k][i];
            }
        }
    }
}

int gate_vpt(int dm)
{
    const int nv = dm / 8;
    const int need = (nv + kBwdThreads - 1) / kBwdThreads;
    return need <= 1 ? 1 : need <= 2 ? 2 : 4;
}

template <typename K>
int64_t wave_blocks(K kernel, int threads, int64_t work)
{
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, 0) != cudaSuccess || per_sm < 1)
        per_sm = 1;
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * per_sm;
    return work < cap ? work : cap;
}

int64_t bwd_blocks(const logo_dims& d, int dm)
{
    const int64_t ntok = static_cast<int64_t>(d.B) * d.T;
    switch (gate_vpt(dm)) {
        case 1: return wave_blocks(gate_bwd_kernel<1>, kBwdThreads, ntok);
        case 2: return wave_blocks(gate_bwd_kernel<2>, kBwdThreads, ntok);
        default: return wave_blocks(gate_bwd_kernel<4>, kBwdThreads, ntok);
    }
}

int check_gate(const logo_dims& d, int dm)
{
    if (d.B < 1 || d.T < 1) return LOGO_ERR_INVALID_ARG;
    if (static_cast<int64_t>(d.B) * d.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    if (dm < 8 || dm % 8 != 0 || dm > kMaxModel) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

}  // namespace
int gate_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" int logo_gate_select(const logo_bf16* x, const float* w_g, int d_model, logo_dims dims, int mode,
                                float b_th, float ratio, float* gate_p, uint8_t* z, int32_t* pos, int32_t* cu_q,
                                int32_t* row_of, int32_t* n_sel_total, void* workspace, size_t workspace_bytes,
                                void* stream)
{
    int rc = check_gate(dims, d_model);
    if (rc != LOGO_OK) return rc;
    if (!x || !w_g || !gate_p || !z || !pos || !cu_q || !row_of || !n_sel_total) return LOGO_ERR_INVALID_ARG;
    if (mode != LOGO_SELECT_THRESHOLD && mode != LOGO_SELECT_RATIO) return LOGO_ERR_INVALID_ARG;
    if (mode == LOGO_SELECT_RATIO && !(ratio >= 0.0f && ratio <= 1.0f)) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(w_g)) return LOGO_ERR_UNSUPPORTED;
    if (!workspace || workspace_bytes < logo_select_workspace_size(dims)) return LOGO_ERR_WORKSPACE;
    const int64_t ntok = static_cast<int64_t>(dims.B) * dims.T;
    const int64_t warps_blocks = (ntok + kFwdThreads / 32 - 1) / (kFwdThreads / 32);
    const unsigned grid = static_cast<unsigned>(wave_blocks(gate_fwd_kernel, kFwdThreads, warps_blocks));
    gate_fwd_kernel<<<grid, kFwdThreads, 0, static_cast<cudaStream_t>(stream)>>>(x, w_g, ntok, d_model, gate_p);
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    return logo_select(gate_p, dims, mode, b_th, ratio, z, pos, cu_q, row_of, n_sel_total, workspace,
                       workspace_bytes, stream);
}

extern "C" size_t logo_gate_bwd_workspace_size(logo_dims dims, int d_model)
{
    if (check_gate(dims, d_model) != LOGO_OK) return 0;
    return static_cast<size_t>(bwd_blocks(dims, d_model)) * static_cast<size_t>(d_model) * sizeof(float);
}

extern "C" int logo_gate_bwd(const logo_bf16* x, const float* w_g, const float* gate_p, const float* dgate_p,
                             int d_model, logo_dims dims, logo_bf16* dx, int accumulate, float* dw_g, void* workspace,
                             size_t workspace_bytes, void* stream)
{
    int rc = check_gate(dims, d_model);
    if (rc != LOGO_OK) return rc;
    if (!x || !w_g || !gate_p || !dgate_p || (!dx && !dw_g)) return LOGO_ERR_INVALID_ARG;
    if (accumulate != 0 && accumulate != 1) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(w_g) || (dx && !aligned16(dx))) return LOGO_ERR_UNSUPPORTED;
    if (dw_g && (!workspace || workspace_bytes < logo_gate_bwd_workspace_size(dims, d_model)))
        return LOGO_ERR_WORKSPACE;
    const int64_t ntok = static_cast<int64_t>(dims.B) * dims.T;
    const unsigned grid = static_cast<unsigned>(bwd_blocks(dims, d_model));
    float* part = dw_g ? static_cast<float*>(workspace) : nullptr;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (gate_vpt(d_model)) {
        case 1: gate_bwd_kernel<1><<<grid, kBwdThreads, 0, st>>>(x, w_g, gate_p, dgate_p, ntok, d_model, dx, accumulate, part); break;
        case 2: gate_bwd_kernel<2><<<grid, kBwdThreads, 0, st>>>(x, w_g, gate_p, dgate_p, ntok, d_model, dx, accumulate, part); break;
        default: gate_bwd_kernel<4><<<grid, kBwdThreads, 0, st>>>(x, w_g, gate_p, dgate_p, ntok, d_model, dx, accumulate, part); break;
    }
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    if (dw_g) {
        colsum_kernel<<<colsum_blocks(d_model), kColSumThreads, 0, st>>>(part, static_cast<int>(grid), d_model, d_model,
                                                                         dw_g, nullptr);
        if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    }
    return LOGO_OK;
}
