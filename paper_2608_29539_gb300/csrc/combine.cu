// combine.cu -- logo_combine / logo_combine_bwd: ContextNorm (Eq. 9, a
// head-wise RMSNorm over D per branch) fused with the gate-weighted output
// fusion of Eq. 10, and the backward of both with z held fixed.
//
// HBM-bound: one block per token; every thread owns 16-byte vectors (8 bf16)
// of one head, the D/8 threads of a head reduce their sums with warp
// shuffles, and the backward reduces dp_t over all heads of the token in
// shared memory.  All arithmetic is fp32; inputs and outputs bf16.
#include <cuda_bf16.h>

#include <cstdint>

#include "host_common.h"
#include "logo_status.cuh"

namespace logo {
namespace {

constexpr int kThreads = 128;

struct Vec8 {
    float v[8];
};

__device__ __forceinline__ Vec8 load_bf16x8(const logo_bf16* p)
{
    uint4 raw = *reinterpret_cast<const uint4*>(p);
    Vec8 r;
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 f = __bfloat1622float2(h[i]);
        r.v[2 * i] = f.x;
        r.v[2 * i + 1] = f.y;
    }
    return r;
}

__device__ __forceinline__ void store_bf16x8(logo_bf16* p, const Vec8& x)
{
    uint4 raw;
    __nv_bfloat162* h = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(x.v[2 * i], x.v[2 * i + 1]);
    *reinterpret_cast<uint4*>(p) = raw;
}

__device__ __forceinline__ Vec8 load_gain(const float* g, int h, int D, int j)
{
    Vec8 r;
    if (g) {
        const float4* p = reinterpret_cast<const float4*>(g + static_cast<int64_t>(h) * D + j * 8);
        float4 a = p[0], b = p[1];
        r.v[0] = a.x; r.v[1] = a.y; r.v[2] = a.z; r.v[3] = a.w;
        r.v[4] = b.x; r.v[5] = b.y; r.v[6] = b.z; r.v[7] = b.w;
    } else {
#pragma unroll
        for (int i = 0; i < 8; ++i) r.v[i] = 1.0f;
    }
    return r;
}

// Sum over the `width` consecutive lanes (a power of two <= 32) of one head.
__device__ __forceinline__ float head_sum(float x, int width)
{
    for (int o = width >> 1; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

__global__ void __launch_bounds__(kThreads) combine_fwd_kernel(
    const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c, const float* __restrict__ gate_p,
    const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of, const float* __restrict__ gain_l,
    const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ o, float* __restrict__ rstd_l,
    float* __restrict__ rstd_g, int H, int D)
{
    const int64_t bt = blockIdx.x;
    const int vpr = D / 8;               // vectors per head row
    const int nvec = H * vpr;            // vectors per token
    const bool sel = z[bt] != 0;
    const int64_t row = sel ? row_of[bt] : -1;
    const float pt = gate_p[bt];
    const float inv_d = 1.0f / static_cast<float>(D);
    for (int v0 = 0; v0 < nvec; v0 += kThreads) {
        const int v = v0 + threadIdx.x;
        const bool active = v < nvec;
        const int h = active ? v / vpr : 0, j = active ? v % vpr : 0;
        Vec8 xl = active ? load_bf16x8(o_l + (bt * H + h) * D + j * 8) : Vec8{};
        float ss = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) ss += xl.v[i] * xl.v[i];
        ss = head_sum(ss, vpr);
        const float rl = rsqrtf(ss * inv_d + eps);
        Vec8 gl = load_gain(gain_l, h, D, j);
        Vec8 out;
#pragma unroll
        for (int i = 0; i < 8; ++i) out.v[i] = xl.v[i] * rl * gl.v[i];
        float rg = 0.f;
        if (sel) {
            Vec8 xg = active ? load_bf16x8(o_c + (row * H + h) * D + j * 8) : Vec8{};
            float sg = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) sg += xg.v[i] * xg.v[i];
            sg = head_sum(sg, vpr);
            rg = rsqrtf(sg * inv_d + eps);
            Vec8 gg = load_gain(gain_g, h, D, j);
#pragma unroll
            for (int i = 0; i < 8; ++i) out.v[i] = (1.0f - pt) * out.v[i] + pt * (xg.v[i] * rg * gg.v[i]);
        }
        if (active) {
            store_bf16x8(o + (bt * H + h) * D + j * 8, out);
            if (j == 0) {
                if (rstd_l) rstd_l[bt * H + h] = rl;
                if (sel && rstd_g) rstd_g[row * H + h] = rg;
            }
        }
    }
}

__global__ void __launch_bounds__(kThreads) combine_bwd_kernel(
    const logo_bf16* __restrict__ dO, const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c,
    const float* __restrict__ gate_p, const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of,
    const float* __restrict__ gain_l, const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ dO_l,
    logo_bf16* __restrict__ dO_c, float* __restrict__ dgate_p, int H, int D)
{
    __shared__ float sh_dp[kThreads / 32];
    const int64_t bt = blockIdx.x;
    const int vpr = D / 8;
    const int nvec = H * vpr;
    const bool sel = z[bt] != 0;
    const int64_t row = sel ? row_of[bt] : -1;
    const float pt = gate_p[bt];
    const float wl = sel ? 1.0f - pt : 1.0f;
    const float inv_d = 1.0f / static_cast<float>(D);
    float dp_acc = 0.f;
    for (int v0 = 0; v0 < nvec; v0 += kThreads) {
        const int v = v0 + threadIdx.x;
        const bool active = v < nvec;
        const int h = active ? v / vpr : 0, j = active ? v % vpr : 0;
        Vec8 g = active ? load_bf16x8(dO + (bt * H + h) * D + j * 8) : Vec8{};
        Vec8 xl = active ? load_bf16x8(o_l + (bt * H + h) * D + j * 8) : Vec8{};
        Vec8 gl = load_gain(gain_l, h, D, j);
        // local branch: dy = dO * wl; dx = r g dy - x r^3 mean(x g dy)
        float ss = 0.f, xgdy = 0.f;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            ss += xl.v[i] * xl.v[i];
            xgdy += xl.v[i] * gl.v[i] * g.v[i];
        }
        ss = head_sum(ss, vpr);
        xgdy = head_sum(xgdy, vpr) * wl;
        const float rl = rsqrtf(ss * inv_d + eps);
        const float cl = rl * rl * rl * xgdy * inv_d;
        Vec8 dxl;
#pragma unroll
        for (int i = 0; i < 8; ++i) dxl.v[i] = rl * gl.v[i] * g.v[i] * wl - xl.v[i] * cl;
        if (active) store_bf16x8(dO_l + (bt * H + h) * D + j * 8, dxl);
        if (sel) {
            Vec8 xg = active ? load_bf16x8(o_c + (row * H + h) * D + j * 8) : Vec8{};
            Vec8 gg = load_gain(gain_g, h, D, j);
            float sg = 0.f, xgdyg = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                sg += xg.v[i] * xg.v[i];
                xgdyg += xg.v[i] * gg.v[i] * g.v[i];
            }
            sg = head_sum(sg, vpr);
            xgdyg = head_sum(xgdyg, vpr) * pt;
            const float rg = rsqrtf(sg * inv_d + eps);
            const float cg = rg * rg * rg * xgdyg * inv_d;
            Vec8 dxg;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                dxg.v[i] = rg * gg.v[i] * g.v[i] * pt - xg.v[i] * cg;
                dp_acc += g.v[i] * (xg.v[i] * rg * gg.v[i] - xl.v[i] * rl * gl.v[i]);
            }
            if (active) store_bf16x8(dO_c + (row * H + h) * D + j * 8, dxg);
        }
    }
    // dp_t = z_t * sum_{h,d} dO (o~G - o~L)
    dp_acc = head_sum(dp_acc, 32);
    if ((threadIdx.x & 31) == 0) sh_dp[threadIdx.x >> 5] = dp_acc;
    __syncthreads();
    if (threadIdx.x == 0) {
        float s = 0.f;
#pragma unroll
        for (int w = 0; w < kThreads / 32; ++w) s += sh_dp[w];
        dgate_p[bt] = sel ? s : 0.0f;
    }
}

int check_combine(const logo_dims& d)
{
    if (d.B < 1 || d.T < 1 || d.Hq < 1) return LOGO_ERR_INVALID_ARG;
    if (d.D != 64 && d.D != 128) return LOGO_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(d.B) * d.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

}  // namespace

int combine_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" int logo_combine(const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p, const uint8_t* z,
                            const int32_t* row_of, const float* gain_l, const float* gain_g, float eps,
                            logo_bf16* o, float* rstd_l, float* rstd_g, logo_dims dims, void* stream)
{
    int rc = check_combine(dims);
    if (rc != LOGO_OK) return rc;
    if (!o_l || !o_c || !gate_p || !z || !row_of || !o) return LOGO_ERR_INVALID_ARG;
    if (!(eps > 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(o_l) || !aligned16(o_c) || !aligned16(o) || (gain_l && !aligned16(gain_l)) ||
        (gain_g && !aligned16(gain_g)))
        return LOGO_ERR_UNSUPPORTED;
    const int64_t ntok = static_cast<int64_t>(dims.B) * dims.T;
    combine_fwd_kernel<<<static_cast<unsigned>(ntok), kThreads, 0, static_cast<cudaStream_t>(stream)>>>(
        o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, o, rstd_l, rstd_g, dims.Hq, dims.D);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

extern "C" int logo_combine_bwd(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p,
                                const uint8_t* z, const int32_t* row_of, const float* gain_l, const float* gain_g,
                                float eps, logo_bf16* dO_l, logo_bf16* dO_c, float* dgate_p, logo_dims dims,
                                void* stream)
{
    int rc = check_combine(dims);
    if (rc != LOGO_OK) return rc;
    if (!dO || !o_l || !o_c || !gate_p || !z || !row_of || !dO_l || !dO_c || !dgate_p) return LOGO_ERR_INVALID_ARG;
    if (!(eps > 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(dO) || !aligned16(o_l) || !aligned16(o_c) || !aligned16(dO_l) || !aligned16(dO_c) ||
        (gain_l && !aligned16(gain_l)) || (gain_g && !aligned16(gain_g)))
        return LOGO_ERR_UNSUPPORTED;
    const int64_t ntok = static_cast<int64_t>(dims.B) * dims.T;
    combine_bwd_kernel<<<static_cast<unsigned>(ntok), kThreads, 0, static_cast<cudaStream_t>(stream)>>>(
        dO, o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, dO_l, dO_c, dgate_p, dims.Hq, dims.D);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
