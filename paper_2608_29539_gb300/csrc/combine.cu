// combine.cu -- logo_combine / logo_combine_bwd(_gains): ContextNorm (Eq. 9,
// a head-wise RMSNorm over D per branch) fused with the gate-weighted output
// fusion of Eq. 10, the backward of both with z held fixed, and the gradients
// of the two ContextNorm gains.
//
// HBM-bound.  Blocks walk the tokens (grid-stride); a thread owns GPT fixed
// groups of G adjacent 16-byte vectors (8 G bf16 of one head row; G = 2 with
// unit gains, 1 when gains are read) of the token's [H, D] row, issues all of
// a token's loads before any arithmetic (so each thread keeps G*GPT to
// 3*G*GPT loads in flight), sums within its group, and the D/(8 G) lanes of a
// head reduce the sums with warp shuffles.  The backward sums dp_t over
// every head of the token in shared memory, and the gain gradients over the
// block's tokens in shared-memory slots that only the thread owning the vector
// touches, then per block into a workspace that a second kernel sums in a
// fixed order (colsum.cuh: deterministic).  All arithmetic is fp32; inputs
// and outputs bf16.
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
constexpr int kMaxVec = 8 * kThreads;   // H*D/8 vectors per token at most (8 vectors per thread)
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
// (branch * 2 + half) * nvec + s holds elements 4 half .. 4 half + 3 of the
// sums of vector v = 2 (s mod npair) + s / npair (s = e npair + u for vector
// e of pair u).  Only the thread that owns the pair touches its slots, and a
// warp's 32 consecutive pairs are 32 consecutive float4 (no bank conflicts).
// In registers they took 32 more per thread (at Hq*D = 4096), which cut the
// resident blocks per SM, and with them the loads in flight, by half.
__device__ __forceinline__ void acc_add8(float4* sh, int nvec, int branch, int s, const Vec8& c)
{
    float4* p0 = sh + (branch * 2) * nvec + s;
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

// A thread owns groups of G adjacent 16-byte vectors of one head row (8 G
// elements).  With G = 2 a head row of D elements is D/16 lanes, so its sums
// take one shuffle level fewer than with a vector per lane and one rsqrt
// serves 16 elements instead of 8: the unit-gain kernels, bound by instruction
// issue as much as by HBM, run with G = 2 when the token row has at least two
// vectors per thread of the block (Hq*D >= 4096: combine 56.7 -> 47.1 us,
// backward 87.9 -> 71.0 us at 16K).  Below that, pairs would leave threads of
// every block idle (4K, Hq*D = 2048: backward 26.5 -> 29.9 us), so G = 1.  The
// kernels that load gains keep G = 1: with two vectors' gains live they
// needed 120-127 registers instead of 72-80.
template <int G>
__device__ __forceinline__ float sumsq_g(const Vec8 (&x)[G])
{
    uint64_t a = 0ull, b = 0ull;
#pragma unroll
    for (int e = 0; e < G; ++e) {
        a = f2_fma(f2_pack(x[e].v[0], x[e].v[1]), f2_pack(x[e].v[0], x[e].v[1]), a);
        b = f2_fma(f2_pack(x[e].v[2], x[e].v[3]), f2_pack(x[e].v[2], x[e].v[3]), b);
        a = f2_fma(f2_pack(x[e].v[4], x[e].v[5]), f2_pack(x[e].v[4], x[e].v[5]), a);
        b = f2_fma(f2_pack(x[e].v[6], x[e].v[7]), f2_pack(x[e].v[6], x[e].v[7]), b);
    }
    float lo, hi;
    f2_unpack(f2_add(a, b), lo, hi);
    return lo + hi;
}

template <int G>
__device__ __forceinline__ float dot_g(const Vec8 (&x)[G], const Vec8 (&y)[G])
{
    uint64_t a = 0ull, b = 0ull;
#pragma unroll
    for (int e = 0; e < G; ++e) {
        a = f2_fma(f2_pack(x[e].v[0], x[e].v[1]), f2_pack(y[e].v[0], y[e].v[1]), a);
        b = f2_fma(f2_pack(x[e].v[2], x[e].v[3]), f2_pack(y[e].v[2], y[e].v[3]), b);
        a = f2_fma(f2_pack(x[e].v[4], x[e].v[5]), f2_pack(y[e].v[4], y[e].v[5]), a);
        b = f2_fma(f2_pack(x[e].v[6], x[e].v[7]), f2_pack(y[e].v[6], y[e].v[7]), b);
    }
    float lo, hi;
    f2_unpack(f2_add(a, b), lo, hi);
    return lo + hi;
}

// dp += dO . (xg r_g - xl r_l) over one vector, as f32x2 pairs
__device__ __forceinline__ uint64_t dp_acc8(uint64_t dp2, const Vec8& g, const Vec8& xl, const Vec8& xg,
                                            uint64_t rl2_neg, uint64_t rg2)
{
#pragma unroll
    for (int i = 0; i < 8; i += 2) {
        const uint64_t t = f2_fma(f2_pack(xl.v[i], xl.v[i + 1]), rl2_neg, f2_mul(f2_pack(xg.v[i], xg.v[i + 1]), rg2));
        dp2 = f2_fma(f2_pack(g.v[i], g.v[i + 1]), t, dp2);
    }
    return dp2;
}

// GPT: groups per thread (group u = vectors G u .. G u + G - 1 of the token's
// [H, D] row; the D/(8 G) lanes of a head reduce its sums with warp shuffles).
template <int GPT, int G, bool UNIT>
__host__ __device__ constexpr int fwd_min_blocks()
{
    return G == 1 && UNIT && GPT == 1 ? 8 : (GPT == 1 || (G == 1 && GPT == 2) ? 5 : 1);
}

template <int GPT, int G, bool UNIT>
__global__ void __launch_bounds__(kThreads, fwd_min_blocks<GPT, G, UNIT>()) combine_fwd_kernel(
    const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c, const float* __restrict__ gate_p,
    const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of, const float* __restrict__ gain_l,
    const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ o, float* __restrict__ rstd_l,
    float* __restrict__ rstd_g, int64_t ntok, int H, int D)
{
    static_assert(G == 1 || (G == 2 && UNIT), "two-vector groups only with unit gains");
    const int vpr = D / 8;               // vectors per head row
    const int gpr = vpr / G;             // groups per head row: the lanes sharing a head
    const int nvec = H * vpr;            // vectors per token
    const int ngrp = nvec / G;
    const float inv_d = 1.0f / static_cast<float>(D);
    for (int64_t bt = blockIdx.x; bt < ntok; bt += gridDim.x) {
        const bool sel = z[bt] != 0;
        const int64_t row = sel ? row_of[bt] : 0;
        const float pt = gate_p[bt];
        uint4 rl[GPT][G], rg[GPT][G];
#pragma unroll
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            const bool active = u < ngrp;
#pragma unroll
            for (int e = 0; e < G; ++e) {
                const int v = G * u + e;
                rl[k][e] = active ? ld_vec(o_l + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
                rg[k][e] = (sel && active) ? ld_vec(o_c + (row * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
            }
        }
#pragma unroll
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            const bool active = u < ngrp;
            const int v0 = G * u;
            const int h = active ? v0 / vpr : 0, j0 = active ? v0 % vpr : 0;
            Vec8 xl[G], out[G];
#pragma unroll
            for (int e = 0; e < G; ++e) xl[e] = unpack8(rl[k][e]);
            float r_l, r_g = 0.f;
            if constexpr (UNIT) {
                r_l = rsqrtf(head_sum(sumsq_g<G>(xl), gpr) * inv_d + eps);
                if (sel) {
                    Vec8 xg[G];
#pragma unroll
                    for (int e = 0; e < G; ++e) xg[e] = unpack8(rg[k][e]);
                    r_g = rsqrtf(head_sum(sumsq_g<G>(xg), gpr) * inv_d + eps);
#pragma unroll
                    for (int e = 0; e < G; ++e) out[e] = axpby8(xl[e], (1.0f - pt) * r_l, &xg[e], pt * r_g);
                } else {
#pragma unroll
                    for (int e = 0; e < G; ++e) out[e] = axpby8(xl[e], r_l, nullptr, 0.f);
                }
            } else {  // G = 1
                float ss = 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) ss += xl[0].v[i] * xl[0].v[i];
                ss = head_sum(ss, gpr);
                r_l = rsqrtf(ss * inv_d + eps);
                const Vec8 gl = load_gain(gain_l, h, D, j0);
#pragma unroll
                for (int i = 0; i < 8; ++i) out[0].v[i] = xl[0].v[i] * r_l * gl.v[i];
                if (sel) {
                    const Vec8 xg = unpack8(rg[k][0]);
                    float sg = 0.f;
#pragma unroll
                    for (int i = 0; i < 8; ++i) sg += xg.v[i] * xg.v[i];
                    sg = head_sum(sg, gpr);
                    r_g = rsqrtf(sg * inv_d + eps);
                    const Vec8 gg = load_gain(gain_g, h, D, j0);
#pragma unroll
                    for (int i = 0; i < 8; ++i) out[0].v[i] = (1.0f - pt) * out[0].v[i] + pt * (xg.v[i] * r_g * gg.v[i]);
                }
            }
            if (active)
#pragma unroll
                for (int e = 0; e < G; ++e) store_bf16x8(o + (bt * nvec + v0 + e) * 8, out[e]);
            if (active && j0 == 0) {
                if (rstd_l) rstd_l[bt * H + h] = r_l;
                if (sel && rstd_g) rstd_g[row * H + h] = r_g;
            }
        }
    }
}

// Register bound of a backward variant: with unit gains one two-vector group
// per thread is held to 4 blocks per SM (3 with the gain sums in shared
// memory), one one-vector group to 5; one-vector groups with the gain sums,
// or with gains read, up to two per thread, are held to 3.
template <int GPT, int G, bool DGAIN, bool UNIT>
__host__ __device__ constexpr int bwd_min_blocks()
{
    return G == 2 ? (GPT == 1 ? (DGAIN ? 3 : 4) : 1)
                  : ((DGAIN || !UNIT) && GPT <= 2 ? 3 : (UNIT && GPT == 1 ? 5 : 1));
}

// part (DGAIN): [gridDim.x][2][H*D] float32 per-block sums of the local and
// global gain gradients, accumulated in dynamic shared memory (4 * nvec float4,
// see acc_add8) over the block's tokens in increasing order.
template <int GPT, int G, bool DGAIN, bool UNIT>
__global__ void __launch_bounds__(kThreads, bwd_min_blocks<GPT, G, DGAIN, UNIT>()) combine_bwd_kernel(
    const logo_bf16* __restrict__ dO, const logo_bf16* __restrict__ o_l, const logo_bf16* __restrict__ o_c,
    const float* __restrict__ gate_p, const uint8_t* __restrict__ z, const int32_t* __restrict__ row_of,
    const float* __restrict__ gain_l, const float* __restrict__ gain_g, float eps, logo_bf16* __restrict__ dO_l,
    logo_bf16* __restrict__ dO_c, float* __restrict__ dgate_p, float* __restrict__ part, int64_t ntok, int H, int D)
{
    static_assert(G == 1 || (G == 2 && UNIT), "two-vector groups only with unit gains");
    __shared__ float sh_dp[2][kThreads / 32];
    const int vpr = D / 8, gpr = vpr / G;
    const int nvec = H * vpr, ngrp = nvec / G;
    const float inv_d = 1.0f / static_cast<float>(D);
    extern __shared__ float4 sh_acc[];
    if (DGAIN) {
#pragma unroll
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            if (u < ngrp)
#pragma unroll
                for (int s = 0; s < 4; ++s)
#pragma unroll
                    for (int e = 0; e < G; ++e) sh_acc[s * nvec + e * ngrp + u] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    int n_sel_seen = 0;
    for (int64_t bt = blockIdx.x; bt < ntok; bt += gridDim.x) {
        const bool sel = z[bt] != 0;
        const int64_t row = sel ? row_of[bt] : 0;
        const float pt = gate_p[bt];
        const float wl = sel ? 1.0f - pt : 1.0f;
        uint4 rd[GPT][G], rl[GPT][G], rg[GPT][G];
#pragma unroll
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            const bool active = u < ngrp;
#pragma unroll
            for (int e = 0; e < G; ++e) {
                const int v = G * u + e;
                rd[k][e] = active ? ld_vec(dO + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
                rl[k][e] = active ? ld_vec(o_l + (bt * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
                rg[k][e] = (sel && active) ? ld_vec(o_c + (row * nvec + v) * 8) : make_uint4(0, 0, 0, 0);
            }
        }
        float dp_acc = 0.f;
        uint64_t dp2 = 0ull;  // UNIT: dp as f32x2 pairs
#pragma unroll
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            const bool active = u < ngrp;
            const int v0 = G * u;
            const int h = active ? v0 / vpr : 0, j0 = active ? v0 % vpr : 0;
            Vec8 g[G], xl[G];
#pragma unroll
            for (int e = 0; e < G; ++e) {
                g[e] = unpack8(rd[k][e]);
                xl[e] = unpack8(rl[k][e]);
            }
            if constexpr (UNIT) {
                // gains 1: dx = r dy - x r^3 mean(x dy), dy = w dO
                const float ss = head_sum(sumsq_g<G>(xl), gpr);
                const float xgdy = head_sum(dot_g<G>(xl, g), gpr) * wl;
                const float r_l = rsqrtf(ss * inv_d + eps);
                const float cl = r_l * r_l * r_l * xgdy * inv_d;
#pragma unroll
                for (int e = 0; e < G; ++e) {
                    if (active) store_bf16x8(dO_l + (bt * nvec + v0 + e) * 8, axpby8(g[e], r_l * wl, &xl[e], -cl));
                    if constexpr (DGAIN) {  // d gain_l = dy * x r
                        Vec8 c;
#pragma unroll
                        for (int i = 0; i < 8; ++i) c.v[i] = g[e].v[i] * wl * xl[e].v[i] * r_l;
                        if (active) acc_add8(sh_acc, nvec, 0, e * ngrp + u, c);
                    }
                }
                if (sel) {
                    Vec8 xg[G];
#pragma unroll
                    for (int e = 0; e < G; ++e) xg[e] = unpack8(rg[k][e]);
                    const float sg = head_sum(sumsq_g<G>(xg), gpr);
                    const float xgdyg = head_sum(dot_g<G>(xg, g), gpr) * pt;
                    const float r_g = rsqrtf(sg * inv_d + eps);
                    const float cg = r_g * r_g * r_g * xgdyg * inv_d;
                    const uint64_t rg2 = f2_pack(r_g, r_g), rl2 = f2_pack(-r_l, -r_l);
#pragma unroll
                    for (int e = 0; e < G; ++e) {
                        if (active) store_bf16x8(dO_c + (row * nvec + v0 + e) * 8, axpby8(g[e], r_g * pt, &xg[e], -cg));
                        if constexpr (DGAIN) {
                            Vec8 c;
#pragma unroll
                            for (int i = 0; i < 8; ++i) c.v[i] = g[e].v[i] * pt * xg[e].v[i] * r_g;
                            if (active) acc_add8(sh_acc, nvec, 1, e * ngrp + u, c);
                        }
                        dp2 = dp_acc8(dp2, g[e], xl[e], xg[e], rl2, rg2);  // dp += dO . (xg r_g - xl r_l)
                    }
                }
                continue;
            }
            // gains read (G = 1): local branch dy = dO * wl; dx = r g dy - x r^3 mean(x g dy)
            const Vec8 gl = load_gain(gain_l, h, D, j0);
            float ss = 0.f, xgdy = 0.f;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                ss += xl[0].v[i] * xl[0].v[i];
                xgdy += xl[0].v[i] * gl.v[i] * g[0].v[i];
            }
            ss = head_sum(ss, gpr);
            xgdy = head_sum(xgdy, gpr) * wl;
            const float r_l = rsqrtf(ss * inv_d + eps);
            const float cl = r_l * r_l * r_l * xgdy * inv_d;
            Vec8 dxl;
#pragma unroll
            for (int i = 0; i < 8; ++i) dxl.v[i] = r_l * gl.v[i] * g[0].v[i] * wl - xl[0].v[i] * cl;
            if (active) store_bf16x8(dO_l + (bt * nvec + v0) * 8, dxl);
            if constexpr (DGAIN) {  // d gain_l = dy * x r
                Vec8 c;
#pragma unroll
                for (int i = 0; i < 8; ++i) c.v[i] = g[0].v[i] * wl * xl[0].v[i] * r_l;
                if (active) acc_add8(sh_acc, nvec, 0, u, c);
            }
            if (sel) {
                const Vec8 xg = unpack8(rg[k][0]);
                const Vec8 gg = load_gain(gain_g, h, D, j0);
                float sg = 0.f, xgdyg = 0.f;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    sg += xg.v[i] * xg.v[i];
                    xgdyg += xg.v[i] * gg.v[i] * g[0].v[i];
                }
                sg = head_sum(sg, gpr);
                xgdyg = head_sum(xgdyg, gpr) * pt;
                const float r_g = rsqrtf(sg * inv_d + eps);
                const float cg = r_g * r_g * r_g * xgdyg * inv_d;
                Vec8 dxg;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    dxg.v[i] = r_g * gg.v[i] * g[0].v[i] * pt - xg.v[i] * cg;
                    dp_acc += g[0].v[i] * (xg.v[i] * r_g * gg.v[i] - xl[0].v[i] * r_l * gl.v[i]);
                }
                if (active) store_bf16x8(dO_c + (row * nvec + v0) * 8, dxg);
                if constexpr (DGAIN) {
                    Vec8 c;
#pragma unroll
                    for (int i = 0; i < 8; ++i) c.v[i] = g[0].v[i] * pt * xg.v[i] * r_g;
                    if (active) acc_add8(sh_acc, nvec, 1, u, c);
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
        for (int k = 0; k < GPT; ++k) {
            const int u = threadIdx.x + k * kThreads;
            if (u < ngrp) {
#pragma unroll
                for (int e = 0; e < G; ++e) {
                    const int v = G * u + e, s = e * ngrp + u;
#pragma unroll
                    for (int br = 0; br < 2; ++br) {
                        float4* dst = reinterpret_cast<float4*>(pl + br * hd + v * 8);
                        dst[0] = sh_acc[(br * 2) * nvec + s];
                        dst[1] = sh_acc[(br * 2 + 1) * nvec + s];
                    }
                }
            }
        }
    }
}

// Vectors per group: two with unit gains when that leaves no thread of the
// block idle (at least 2 x kThreads vectors per token), else one.
int group_vectors(const logo_dims& d, bool unit)
{
    return unit && d.Hq * (d.D / 8) >= 2 * kThreads ? 2 : 1;
}

// Groups of vectors per thread: 1, 2, 4 or 8.
int groups_per_thread(const logo_dims& d, int g)
{
    const int ngrp = d.Hq * (d.D / 8) / g;
    const int need = (ngrp + kThreads - 1) / kThreads;
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
    int64_t with_gains = 0, unit = 0;
    switch (groups_per_thread(d, 1)) {
        case 1:
            gains_smem_ok(combine_bwd_kernel<1, 1, true, false>);
            with_gains = wave_blocks(combine_bwd_kernel<1, 1, true, false>, ntok, smem);
            break;
        case 2:
            gains_smem_ok(combine_bwd_kernel<2, 1, true, false>);
            with_gains = wave_blocks(combine_bwd_kernel<2, 1, true, false>, ntok, smem);
            break;
        default:
            gains_smem_ok(combine_bwd_kernel<4, 1, true, false>);
            with_gains = wave_blocks(combine_bwd_kernel<4, 1, true, false>, ntok, smem);
            break;
    }
    const int gu = group_vectors(d, true), gpt = groups_per_thread(d, gu);
    if (gu == 1) {
        gains_smem_ok(combine_bwd_kernel<1, 1, true, true>);
        unit = wave_blocks(combine_bwd_kernel<1, 1, true, true>, ntok, smem);
    } else if (gpt == 1) {
        gains_smem_ok(combine_bwd_kernel<1, 2, true, true>);
        unit = wave_blocks(combine_bwd_kernel<1, 2, true, true>, ntok, smem);
    } else {
        gains_smem_ok(combine_bwd_kernel<2, 2, true, true>);
        unit = wave_blocks(combine_bwd_kernel<2, 2, true, true>, ntok, smem);
    }
    return std::max(with_gains, unit);
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
#define LOGO_COMBINE_FWD(V, G, U)                                                                           \
    combine_fwd_kernel<V, G, U><<<static_cast<unsigned>(wave_blocks(combine_fwd_kernel<V, G, U>, ntok)), kThreads, \
                                  0, st>>>(o_l, o_c, gate_p, z, row_of, gain_l, gain_g, eps, o, rstd_l, rstd_g,      \
                                           ntok, dims.Hq, dims.D)
    const bool unit = !gain_l && !gain_g;
    const int g = group_vectors(dims, unit), gpt = groups_per_thread(dims, g);
    if (g == 2) {
        switch (gpt) {
            case 1: LOGO_COMBINE_FWD(1, 2, true); break;
            case 2: LOGO_COMBINE_FWD(2, 2, true); break;
            default: LOGO_COMBINE_FWD(4, 2, true); break;
        }
    } else if (unit) {  // fewer than 2 x kThreads vectors a token
        if (gpt == 1) { LOGO_COMBINE_FWD(1, 1, true); }
        else { LOGO_COMBINE_FWD(2, 1, true); }
    } else {
        switch (gpt) {
            case 1: LOGO_COMBINE_FWD(1, 1, false); break;
            case 2: LOGO_COMBINE_FWD(2, 1, false); break;
            case 4: LOGO_COMBINE_FWD(4, 1, false); break;
            default: LOGO_COMBINE_FWD(8, 1, false); break;
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
    const bool unit = !gain_l && !gain_g;
    const int g = group_vectors(dims, unit), gpt = groups_per_thread(dims, g);
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
#define LOGO_COMBINE_BWD(V, NV, GN, U)                                                                          \
    if (GN && !gains_smem_ok(combine_bwd_kernel<V, NV, GN, U>)) return LOGO_ERR_CUDA;                             \
    grid = static_cast<unsigned>(wave_blocks(combine_bwd_kernel<V, NV, GN, U>, ntok, smem));                      \
    combine_bwd_kernel<V, NV, GN, U><<<grid, kThreads, smem, st>>>(dO, o_l, o_c, gate_p, z, row_of, gain_l, gain_g,   \
                                                                   eps, dO_l, dO_c, dgate_p, part, ntok, dims.Hq,    \
                                                                   dims.D)
    if (gains && unit) {
        if (g == 1) { LOGO_COMBINE_BWD(1, 1, true, true); }
        else if (gpt == 1) { LOGO_COMBINE_BWD(1, 2, true, true); }
        else { LOGO_COMBINE_BWD(2, 2, true, true); }
    } else if (gains) {
        switch (gpt) {
            case 1: LOGO_COMBINE_BWD(1, 1, true, false); break;
            case 2: LOGO_COMBINE_BWD(2, 1, true, false); break;
            default: LOGO_COMBINE_BWD(4, 1, true, false); break;
        }
    } else if (unit && g == 2) {
        switch (gpt) {
            case 1: LOGO_COMBINE_BWD(1, 2, false, true); break;
            case 2: LOGO_COMBINE_BWD(2, 2, false, true); break;
            default: LOGO_COMBINE_BWD(4, 2, false, true); break;
        }
    } else if (unit) {  // fewer than 2 x kThreads vectors a token
        if (gpt == 1) { LOGO_COMBINE_BWD(1, 1, false, true); }
        else { LOGO_COMBINE_BWD(2, 1, false, true); }
    } else {
        switch (gpt) {
            case 1: LOGO_COMBINE_BWD(1, 1, false, false); break;
            case 2: LOGO_COMBINE_BWD(2, 1, false, false); break;
            case 4: LOGO_COMBINE_BWD(4, 1, false, false); break;
            default: LOGO_COMBINE_BWD(8, 1, false, false); break;
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
