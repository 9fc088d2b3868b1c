// combine.cu -- logo_combine / logo_combine_bwd(_gains): ContextNorm (Eq. 9,
// a head-wise RMSNorm over D per branch) fused with the gate-weighted output
// fusion of Eq. 10, the backward of both with z held fixed, and the gradients
// of the two ContextNorm gains.
//
// HBM-bound.  Blocks walk the tokens (grid-stride); a thread owns VPT fixed
// 16-byte vectors (8 bf16) of the token's [H, D] row, issues all of a token's
// loads before any arithmetic (so each thread keeps VPT to 3*VPT loads in
// flight), and the D/8 lanes of a head reduce their sums with warp shuffles.
// The backward sums dp_t over every head of the token in shared memory, and
// the gain gradients over the block's tokens in shared-memory slots that only
// the thread owning the vector touches, then per block into a workspace that a
// second kernel sums in a fixed order (colsum.cuh: deterministic).  All arithmetic is fp32; inputs and outputs bf16.
// The kernels are bound as much by instruction issue as by HBM: without gains
// (both NULL, i.e. 1) a separate instantiation drops the gain loads and the
// unit multiplies and does the elementwise work as f32x2 pairs.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>

#include "colsum.cuh"
#include "host_common.h"
#include "logo_status.cuh"
#include "sm100.cuh"

namespace logo {
namespace {

constexpr int kThreads = 256;
constexpr int kMaxVec = 8 * kThreads;   // H*D/8 vectors per token at most (VPT <= 8)
constexpr int kMaxVecGains = 4 * kThreads;

struct Vec8 {
    float v[8];
};

__device__ __forceinline__ uint4 ld_vec(const logo_bf16* p) { return *reinterpret_cast<const uint4*>(p); }

__device__ __forceinline__ Vec8 unpack8(const uint4& raw)
{
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

// sum_i x_i^2 and sum_i x_i y_i over a vector of 8, as f32x2 pairs
__device__ __forceinline__ float sumsq8(const Vec8& x)
{
    uint64_t a = f2_mul(f2_pack(x.v[0], x.v[1]), f2_pack(x.v[0], x.v[1]));
    uint64_t b = f2_mul(f2_pack(x.v[2], x.v[3]), f2_pack(x.v[2], x.v[3]));
    a = f2_fma(f2_pack(x.v[4], x.v[5]), f2_pack(x.v[4], x.v[5]), a);
    b = f2_fma(f2_pack(x.v[6], x.v[7]), f2_pack(x.v[6], x.v[7]), b);
    float lo, hi;
    f2_unpack(f2_add(a, b), lo, hi);
    return lo + hi;
}

__device__ __forceinline__ float dot8(const Vec8& x, const Vec8& y)
{
    uint64_t a = f2_mul(f2_pack(x.v[0], x.v[1]), f2_pack(y.v[0], y.v[1]));
    uint64_t b = f2_mul(f2_pack(x.v[2], x.v[3]), f2_pack(y.v[2], y.v[3]));
    a = f2_fma(f2_pack(x.v[4], x.v[5]), f2_pack(y.v[4], y.v[5]), a);
    b = f2_fma(f2_pack(x.v[6], x.v[7]), f2_pack(y.v[6], y.v[7]), b);
    float lo, hi;
    f2_unpack(f2_add(a, b), lo, hi);
    return lo + hi;
}

// x * a + y * b elementwise (y, b optional), as f32x2 pairs
__device__ __forceinline__ Vec8 axpby8(const Vec8& x, float a, const Vec8* y, float b)
{
    const uint64_t a2 = f2_pack(a, a), b2 = f2_pack(b, b);
    Vec8 r;
#pragma unroll
    for (int i = 0; i < 8; i += 2) {
        uint64_t t = f2_mul(f2_pack(x.v[i], x.v[i + 1]), a2);
        if (y) t = f2_fma(f2_pack(y->v[i], y->v[i + 1]), b2, t);
        f2_unpack(t, r.v[i], r.v[i + 1]);
    }
    return r;
}

// Gain-gradient accumulators of the backward, in shared memory: float4 slot
// (branch * 2 + half) * nvec + v holds elements 4 half .. 4 half + 3 of vector
// v's sums.  Only the thread that owns vector v touches its slots, and a
// warp's 32 consecutive vectors are 32 consecutive float4 (no bank conflicts).
// In registers they took 32 more per thread (at Hq*D = 4096), which cut the
// resident blocks per SM, and with them the loads in flight, by half.
__device__ __forceinline__ void acc_add8(float4* sh, int nvec, int branch, int v, const Vec8& c)
{
    float4* p0 = sh + (branch * 2) * nvec + v;
    float4* p1 = p0 + nvec;
    float4 a = *p0, b = *p1;
    a.x += c.v[0]; a.y += c.v[1]; a.z += c.v[2]; a.w += c.v[3];
    b.x += c.v[4]; b.y += c.v[5]; b.z += c.v[6]; b.w += c.v[7];
    *p0 = a;
    *p1 = b;
}

// Sum over the `width` consecutive lanes (a power of two <= 32) of one head.
__device__ __forceinline__ float head_sum(float x, int width)
{
    for (int o = width >> 1; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
    return x;
}

template <int VPT, bool UNIT>
__global__ void __launch_bounds__(kThreads) combine_fwd_kernel(
    const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c, const float* __restrict__ gate_p,
    const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of, const float* __restrict__ gain_l,
    const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ o, float* __restrict__ rstd_l,
    float* __restrict__ rstd_g, int64_t ntok, int H, int D)
{
    const int vpr = D / 8;               // vectors per head row
    const int nvec = H * vpr;            // vectors per token
    const float inv_d = 1.0f / static_cast<float>(D);
    for (int64_t bt = blockIdx.x; bt < ntok; bt += gridDim.x) {
        const bool sel = z[bt] != 0;
        const int64_t row = sel ? row_of[bt] : 0;
        const float pt = gate_p[bt];
        uint4 rl[VPT], rg[VPT];
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            rl[k] = v < nvec ? ld_vec(o_l + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
            rg[k] = (sel && v < nvec) ? ld_vec(o_c + (row * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            const bool active = v < nvec;
            const int h = active ? v / vpr : 0, j = active ? v % vpr : 0;
            const Vec8 xl = unpack8(rl[k]);
            Vec8 out;
            float r_l, r_g = 0.f;
            if constexpr (UNIT) {
                r_l = rsqrtf(head_sum(sumsq8(xl), vpr) * inv_d + eps);
                if (sel) {
                    const Vec8 xg = unpack8(rg[k]);
                    r_g = rsqrtf(head_sum(sumsq8(xg), vpr) * inv_d + eps);
                    out = axpby8(xl, (1.0f - pt) * r_l, &xg, pt * r_g);
                } else {
                    out = axpby8(xl, r_l, nullptr, 0.f);
                }
            } else {
            float ss = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) ss += xl.v[i] * xl.v[i];
            ss = head_sum(ss, vpr);
            r_l = rsqrtf(ss * inv_d + eps);
            const Vec8 gl = load_gain(gain_l, h, D, j);
#pragma unroll
            for (int i = 0; i < 8; ++i) out.v[i] = xl.v[i] * r_l * gl.v[i];
            if (sel) {
                const Vec8 xg = unpack8(rg[k]);
                float sg = 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) sg += xg.v[i] * xg.v[i];
                sg = head_sum(sg, vpr);
                r_g = rsqrtf(sg * inv_d + eps);
                const Vec8 gg = load_gain(gain_g, h, D, j);
#pragma unroll
                for (int i = 0; i < 8; ++i) out.v[i] = (1.0f - pt) * out.v[i] + pt * (xg.v[i] * r_g * gg.v[i]);
            }
            }
            if (active) {
                store_bf16x8(o + (bt * nvec + v) * 8, out);
                if (j == 0) {
                    if (rstd_l) rstd_l[bt * H + h] = r_l;
                    if (sel && rstd_g) rstd_g[row * H + h] = r_g;
                }
            }
        }
    }
}

// part (DGAIN): [gridDim.x][2][H*D] float32 per-block sums of the local and
// global gain gradients, accumulated in dynamic shared memory (4 * nvec float4,
// see acc_add8) over the block's tokens in increasing order.
template <int VPT, bool DGAIN, bool UNIT>
__global__ void __launch_bounds__(kThreads, DGAIN && VPT <= 2 ? 3 : 1) combine_bwd_kernel(
    const logo_bf16* __restrict__ dO, const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c,
    const float* __restrict__ gate_p, const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of,
    const float* __restrict__ gain_l, const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ dO_l,
    logo_bf16* __restrict__ dO_c, float* __restrict__ dgate_p, float* __restrict__ part, int64_t ntok, int H, int D)
{
    __shared__ float sh_dp[2][kThreads / 32];
    const int vpr = D / 8;
    const int nvec = H * vpr;
    const float inv_d = 1.0f / static_cast<float>(D);
    extern __shared__ float4 sh_acc[];
    if (DGAIN) {
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            if (v < nvec)
#pragma unroll
                for (int s = 0; s < 4; ++s) sh_acc[s * nvec + v] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    int n_sel_seen = 0;
    for (int64_t bt = blockIdx.x; bt < ntok; bt += gridDim.x) {
        const bool sel = z[bt] != 0;
        const int64_t row = sel ? row_of[bt] : 0;
        const float pt = gate_p[bt];
        const float wl = sel ? 1.0f - pt : 1.0f;
        uint4 rd[VPT], rl[VPT], rg[VPT];
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            const bool active = v < nvec;
            rd[k] = active ? ld_vec(dO + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
            rl[k] = active ? ld_vec(o_l + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
            rg[k] = (sel && active) ? ld_vec(o_c + (row * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
        }
        float dp_acc = 0.f;
        uint64_t dp2 = 0ull;  // UNIT: dp as f32x2 pairs
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            const bool active = v < nvec;
            const int h = active ? v / vpr : 0, j = active ? v % vpr : 0;
            const Vec8 g = unpack8(rd[k]);
            const Vec8 xl = unpack8(rl[k]);
            if constexpr (UNIT) {
                // gains 1: dx = r dy - x r^3 mean(x dy), dy = w dO
                const float ss = head_sum(sumsq8(xl), vpr);
                const float xgdy = head_sum(dot8(xl, g), vpr) * wl;
                const float r_l = rsqrtf(ss * inv_d + eps);
                const float cl = r_l * r_l * r_l * xgdy * inv_d;
                if (active) store_bf16x8(dO_l + (bt * nvec + v) * 8, axpby8(g, r_l * wl, &xl, -cl));
                if constexpr (DGAIN) {  // d gain_l = dy * x r
                    Vec8 c;
#pragma unroll
                    for (int i = 0; i < 8; ++i) c.v[i] = g.v[i] * wl * xl.v[i] * r_l;
                    if (active) acc_add8(sh_acc, nvec, 0, v, c);
                }
                if (sel) {
                    const Vec8 xg = unpack8(rg[k]);
                    const float sg = head_sum(sumsq8(xg), vpr);
                    const float xgdyg = head_sum(dot8(xg, g), vpr) * pt;
                    const float r_g = rsqrtf(sg * inv_d + eps);
                    const float cg = r_g * r_g * r_g * xgdyg * inv_d;
                    if (active) store_bf16x8(dO_c + (row * nvec + v) * 8, axpby8(g, r_g * pt, &xg, -cg));
                    if constexpr (DGAIN) {
                        Vec8 c;
#pragma unroll
                        for (int i = 0; i < 8; ++i) c.v[i] = g.v[i] * pt * xg.v[i] * r_g;
                        if (active) acc_add8(sh_acc, nvec, 1, v, c);
                    }
                    // dp += dO . (xg r_g - xl r_l)
                    const uint64_t rg2 = f2_pack(r_g, r_g), rl2 = f2_pack(-r_l, -r_l);
#pragma unroll
                    for (int i = 0; i < 8; i += 2) {
                        const uint64_t t = f2_fma(f2_pack(xl.v[i], xl.v[i + 1]), rl2,
                                                  f2_mul(f2_pack(xg.v[i], xg.v[i + 1]), rg2));
                        dp2 = f2_fma(f2_pack(g.v[i], g.v[i + 1]), t, dp2);
                    }
                }
                continue;
            }
            const Vec8 gl = load_gain(gain_l, h, D, j);
            // local branch: dy = dO * wl; dx = r g dy - x r^3 mean(x g dy)
            float ss = 0.f, xgdy = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                ss += xl.v[i] * xl.v[i];
                xgdy += xl.v[i] * gl.v[i] * g.v[i];
            }
            ss = head_sum(ss, vpr);
            xgdy = head_sum(xgdy, vpr) * wl;
            const float r_l = rsqrtf(ss * inv_d + eps);
            const float cl = r_l * r_l * r_l * xgdy * inv_d;
            Vec8 dxl;
#pragma unroll
            for (int i = 0; i < 8; ++i) dxl.v[i] = r_l * gl.v[i] * g.v[i] * wl - xl.v[i] * cl;
            if (active) store_bf16x8(dO_l + (bt * nvec + v) * 8, dxl);
            if constexpr (DGAIN) {  // d gain_l = dy * x r
                Vec8 c;
#pragma unroll
                for (int i = 0; i < 8; ++i) c.v[i] = g.v[i] * wl * xl.v[i] * r_l;
                if (active) acc_add8(sh_acc, nvec, 0, v, c);
            }
            if (sel) {
                const Vec8 xg = unpack8(rg[k]);
                const Vec8 gg = load_gain(gain_g, h, D, j);
                float sg = 0.f, xgdyg = 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    sg += xg.v[i] * xg.v[i];
                    xgdyg += xg.v[i] * gg.v[i] * g.v[i];
                }
                sg = head_sum(sg, vpr);
                xgdyg = head_sum(xgdyg, vpr) * pt;
                const float r_g = rsqrtf(sg * inv_d + eps);
                const float cg = r_g * r_g * r_g * xgdyg * inv_d;
                Vec8 dxg;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    dxg.v[i] = r_g * gg.v[i] * g.v[i] * pt - xg.v[i] * cg;
                    dp_acc += g.v[i] * (xg.v[i] * r_g * gg.v[i] - xl.v[i] * r_l * gl.v[i]);
                }
                if (active) store_bf16x8(dO_c + (row * nvec + v) * 8, dxg);
                if constexpr (DGAIN) {
                    Vec8 c;
#pragma unroll
                    for (int i = 0; i < 8; ++i) c.v[i] = g.v[i] * pt * xg.v[i] * r_g;
                    if (active) acc_add8(sh_acc, nvec, 1, v, c);
                }
            }
        }
        if constexpr (UNIT) {
            float lo, hi;
            f2_unpack(dp2, lo, hi);
            dp_acc = lo + hi;
        }
        // dp_t = z_t * sum_{h,d} dO (o~G - o~L); z_t is uniform over the block
        if (sel) {
            const int buf = n_sel_seen & 1;
            ++n_sel_seen;
            dp_acc = head_sum(dp_acc, 32);
            if ((threadIdx.x & 31) == 0) sh_dp[buf][threadIdx.x >> 5] = dp_acc;
            __syncthreads();
            if (threadIdx.x == 0) {
                float s = 0.f;
#pragma unroll
                for (int w = 0; w < kThreads / 32; ++w) s += sh_dp[buf][w];
                dgate_p[bt] = s;
            }
        } else if (threadIdx.x == 0) {
            dgate_p[bt] = 0.0f;
        }
    }
    if (DGAIN) {
        const int64_t hd = static_cast<int64_t>(nvec) * 8;
        float* pl = part + static_cast<int64_t>(blockIdx.x) * 2 * hd;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * kThreads;
            if (v < nvec) {
#pragma unroll
                for (int br = 0; br < 2; ++br) {
                    float4* dst = reinterpret_cast<float4*>(pl + br * hd + v * 8);
                    dst[0] = sh_acc[(br * 2) * nvec + v];
                    dst[1] = sh_acc[(br * 2 + 1) * nvec + v];
                }
            }
        }
    }
}

int vec_per_thread(const logo_dims& d)
{
    const int nvec = d.Hq * (d.D / 8);
    const int need = (nvec + kThreads - 1) / kThreads;
    return need <= 1 ? 1 : need <= 2 ? 2 : need <= 4 ? 4 : 8;
}

// One wave of resident blocks (the grid-stride loop gives every block the
// same number of tokens), capped by the token count.
template <typename K>
int64_t wave_blocks(K kernel, int64_t ntok, size_t smem = 0)
{
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kThreads, smem) != cudaSuccess || per_sm < 1)
        per_sm = 1;
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * per_sm;
    return ntok < cap ? ntok : cap;
}

// Dynamic shared memory of the gain-gradient backward: its accumulators.
size_t gains_smem(const logo_dims& d) { return static_cast<size_t>(4) * (d.Hq * d.D / 8) * sizeof(float4); }

// The gain variant may need more than the default 48 KB of dynamic shared
// memory (64 KB at Hq*D = 8192); the attribute is set before any occupancy
// query or launch of it.
template <typename K>
bool gains_smem_ok(K kernel)
{
    return set_smem_limit(kernel, 4 * kMaxVecGains * static_cast<int>(sizeof(float4))) == cudaSuccess;
}

// Blocks of the gain-gradient backward (one partial row each): the larger of
// its two variants, so the workspace fits whichever runs.
int64_t gains_blocks(const logo_dims& d)
{
    const int64_t ntok = static_cast<int64_t>(d.B) * d.T;
    const size_t smem = gains_smem(d);
    switch (vec_per_thread(d)) {
        case 1:
            gains_smem_ok(combine_bwd_kernel<1, true, false>);
            gains_smem_ok(combine_bwd_kernel<1, true, true>);
            return std::max(wave_blocks(combine_bwd_kernel<1, true, false>, ntok, smem),
                            wave_blocks(combine_bwd_kernel<1, true, true>, ntok, smem));
        case 2:
            gains_smem_ok(combine_bwd_kernel<2, true, false>);
            gains_smem_ok(combine_bwd_kernel<2, true, true>);
            return std::max(wave_blocks(combine_bwd_kernel<2, true, false>, ntok, smem),
                            wave_blocks(combine_bwd_kernel<2, true, true>, ntok, smem));
        default:
            gains_smem_ok(combine_bwd_kernel<4, true, false>);
            gains_smem_ok(combine_bwd_kernel<4, true, true>);
            return std::max(wave_blocks(combine_bwd_kernel<4, true, false>, ntok, smem),
                            wave_blocks(combine_bwd_kernel<4, true, true>, ntok, smem));
    }
}

int check_combine(const logo_dims& d)
{
    if (d.B < 1 || d.T < 1 || d.Hq < 1) return LOGO_ERR_INVALID_ARG;
    if (d.D != 64 && d.D != 128) return LOGO_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(d.B) * d.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    if (d.Hq * (d.D / 8) > kMaxVec) return LOGO_ERR_UNSUPPORTED;  // Hq * D <= 16384
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
    cudaStream_t st = static_cast<cudaStream_t>(stream);
#define LOGO_COMBINE_FWD(V, U)                                                                                 \
    combine_fwd_kernel<V, U><<<static_cast<unsigned>(wave_blocks(combine_fwd_kernel<V, U>, ntok)), kThreads, 0, \
                               st>>>(o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, o, rstd_l, rstd_g, ntok,    \
                                     dims.Hq, dims.D)
    if (!gain_l && !gain_g) {
        switch (vec_per_thread(dims)) {
            case 1: LOGO_COMBINE_FWD(1, true); break;
            case 2: LOGO_COMBINE_FWD(2, true); break;
            case 4: LOGO_COMBINE_FWD(4, true); break;
            default: LOGO_COMBINE_FWD(8, true); break;
        }
    } else {
        switch (vec_per_thread(dims)) {
            case 1: LOGO_COMBINE_FWD(1, false); break;
            case 2: LOGO_COMBINE_FWD(2, false); break;
            case 4: LOGO_COMBINE_FWD(4, false); break;
            default: LOGO_COMBINE_FWD(8, false); break;
        }
    }
#undef LOGO_COMBINE_FWD
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

namespace {
int combine_bwd_common(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p,
                       const uint8_t* z, const int32_t* row_of, const float* gain_l, const float* gain_g, float eps,
                       logo_bf16* dO_l, logo_bf16* dO_c, float* dgate_p, float* dgain_l, float* dgain_g,
                       void* workspace, size_t workspace_bytes, logo_dims dims, void* stream)
{
    int rc = check_combine(dims);
    if (rc != LOGO_OK) return rc;
    if (!dO || !o_l || !o_c || !gate_p || !z || !row_of || !dO_l || !dO_c || !dgate_p) return LOGO_ERR_INVALID_ARG;
    if (!(eps > 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(dO) || !aligned16(o_l) || !aligned16(o_c) || !aligned16(dO_l) || !aligned16(dO_c) ||
        (gain_l && !aligned16(gain_l)) || (gain_g && !aligned16(gain_g)))
        return LOGO_ERR_UNSUPPORTED;
    const bool gains = dgain_l || dgain_g;
    const int vpt = vec_per_thread(dims);
    if (gains) {
        if (dims.Hq * (dims.D / 8) > kMaxVecGains) return LOGO_ERR_UNSUPPORTED;  // Hq * D <= 8192
        if (!workspace) return LOGO_ERR_INVALID_ARG;
        if (workspace_bytes < logo_combine_bwd_workspace_size(dims)) return LOGO_ERR_WORKSPACE;
    }
    const int64_t ntok = static_cast<int64_t>(dims.B) * dims.T;
    const size_t smem = gains ? gains_smem(dims) : 0;
    unsigned grid = 0;
    float* part = static_cast<float*>(workspace);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
#define LOGO_COMBINE_BWD(V, G, U)                                                                                 \
    if (G && !gains_smem_ok(combine_bwd_kernel<V, G, U>)) return LOGO_ERR_CUDA;                                    \
    grid = static_cast<unsigned>(wave_blocks(combine_bwd_kernel<V, G, U>, ntok, smem));                            \
    combine_bwd_kernel<V, G, U><<<grid, kThreads, smem, st>>>(dO, o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps,    \
                                                              dO_l, dO_c, dgate_p, part, ntok, dims.Hq, dims.D)
    const bool unit = !gain_l && !gain_g;
    if (gains && unit) {
        switch (vpt) {
            case 1: LOGO_COMBINE_BWD(1, true, true); break;
            case 2: LOGO_COMBINE_BWD(2, true, true); break;
            default: LOGO_COMBINE_BWD(4, true, true); break;
        }
    } else if (gains) {
        switch (vpt) {
            case 1: LOGO_COMBINE_BWD(1, true, false); break;
            case 2: LOGO_COMBINE_BWD(2, true, false); break;
            default: LOGO_COMBINE_BWD(4, true, false); break;
        }
    } else if (unit) {
        switch (vpt) {
            case 1: LOGO_COMBINE_BWD(1, false, true); break;
            case 2: LOGO_COMBINE_BWD(2, false, true); break;
            case 4: LOGO_COMBINE_BWD(4, false, true); break;
            default: LOGO_COMBINE_BWD(8, false, true); break;
        }
    } else {
        switch (vpt) {
            case 1: LOGO_COMBINE_BWD(1, false, false); break;
            case 2: LOGO_COMBINE_BWD(2, false, false); break;
            case 4: LOGO_COMBINE_BWD(4, false, false); break;
            default: LOGO_COMBINE_BWD(8, false, false); break;
        }
    }
#undef LOGO_COMBINE_BWD
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    if (gains) {
        const int hd = dims.Hq * dims.D;
        colsum_kernel<<<colsum_blocks(2 * hd), kColSumThreads, 0, st>>>(part, static_cast<int>(grid), 2 * hd, hd,
                                                                        dgain_l, dgain_g);
        if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    }
    return LOGO_OK;
}
}  // namespace

extern "C" int logo_combine_bwd(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p,
                                const uint8_t* z, const int32_t* row_of, const float* gain_l, const float* gain_g,
                                float eps, logo_bf16* dO_l, logo_bf16* dO_c, float* dgate_p, logo_dims dims,
                                void* stream)
{
    return combine_bwd_common(dO, o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, dO_l, dO_c, dgate_p, nullptr,
                              nullptr, nullptr, 0, dims, stream);
}

extern "C" size_t logo_combine_bwd_workspace_size(logo_dims dims)
{
    if (check_combine(dims) != LOGO_OK) return 0;
    if (dims.Hq * (dims.D / 8) > kMaxVecGains) return 0;
    return static_cast<size_t>(gains_blocks(dims)) * 2 * static_cast<size_t>(dims.Hq) * dims.D * sizeof(float);
}

extern "C" int logo_combine_bwd_gains(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c,
                                      const float* gate_p, const uint8_t* z, const int32_t* row_of,
                                      const float* gain_l, const float* gain_g, float eps, logo_bf16* dO_l,
                                      logo_bf16* dO_c, float* dgate_p, float* dgain_l, float* dgain_g,
                                      logo_dims dims, void* workspace, size_t workspace_bytes, void* stream)
{
    if (!dgain_l && !dgain_g) return LOGO_ERR_INVALID_ARG;
    return combine_bwd_common(dO, o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, dO_l, dO_c, dgate_p, dgain_l,
                              dgain_g, workspace, workspace_bytes, dims, stream);
}
