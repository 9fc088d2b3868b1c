// attn_bwd.cu -- backward of both attention branches on tcgen05 tensor cores.
//
//   logo_local_attn_bwd          gradients of Eq. 6 (window W, every token)
//   logo_global_sparse_attn_bwd  row-sparse gradients of Eq. 8 (Sec. 3.3, App. B)
//
// With P = softmax(scale * Q K^T) over the visible keys, dO the upstream
// gradient and Dsum = rowsum(dO * O):
//   dV = P^T dO,  dP = dO V^T,  dS = P * (dP - Dsum),
//   dQ = scale * dS K,  dK = scale * dS^T Q.
// Both kernels are persistent and KV-block-major: a work item is one block of
// 128 keys of one KV head of one sequence, and it walks every (query head of
// the KV head's group) x (query tile that can see the block).  dK and dV stay
// in TMEM for the whole item (one CTA owns the block for every query head of
// its group, so they need no atomics); dQ is reduced across items in fp32.
// Five MMAs per (query tile, KV block), the minimum: the paper's separate dQ
// and dK/dV kernels recompute S and dP and take seven.
//
// d = 128, attn_bwd2_kernel (16 warps, query tiles of 64 rows):
//   warp 0       TMA: K/V once per item, Q/dO tiles through a 4-deep ring
//   warp 1       MMA issuer A: S^T = K Q^T, dP^T = V dO^T (M = 128 keys,
//                N = 64 queries) into one TMEM buffer that the softmax warps
//                release as soon as they have loaded it
//   warps 2..9   two warpgroups, one per 32-query half of the tile; thread =
//                key row: P^T (back to TMEM as bf16 pairs, two buffers) and
//                dS^T (bf16, to shared memory, two buffers)
//   warp 15      MMA issuer B: dV += P^T dO (P^T as the TMEM operand),
//                dK += dS^T Q, dQ^T = K^T dS^T into a TMEM buffer of its own
//   warps 10..13 dQ^T out of TMEM (thread = head-dim row), coalesced fp32
//                reductions into the dQ accumulator (one 128-byte row segment
//                per warp instruction), converted to bf16 by a pass after the
//                kernel; dK/dV epilogue at the end of each item
//   warp 14      global branch: zero rows of the dense dQ for unselected tokens
// Global query tiles are 64-row slices of the packed selected rows, starting
// at the first packed row whose position reaches the block, read from a table
// the pre-pass builds once per call (App. B's precomputed search); the same
// pre-pass gathers the selected Q rows and computes Dsum.
//
// d = 64, attn_bwd_kernel (6 warps, query tiles of 128 rows): one MMA warp
// issues S^T, dP^T, then dV, dK and dQ into the S^T columns once the softmax
// warps have written P^T and dS^T to shared memory; the first visible query
// tile of a global item comes from a binary search over the packed positions;
// dQ goes through fp32 atomics and a conversion pass.
#include <cuda_bf16.h>

#include <cstdint>
#include <type_traits>

#include "attn_common.cuh"
#include "host_common.h"
#include "sm100.cuh"

namespace logo {
namespace {

template <int D>
struct BwdCfg {
    static constexpr int kSub = D / 64;
    static constexpr int kTileBytes = kBM * D * 2;
    static constexpr int kOffK = 0;
    static constexpr int kOffV = kOffK + kTileBytes;
    static constexpr int kOffQ = kOffV + kTileBytes;
    static constexpr int kOffDO = kOffQ + kTileBytes;
    static constexpr int kOffP = kOffDO + kTileBytes;     // P^T  [128 keys][128 queries] bf16
    static constexpr int kOffDS = kOffP + kBM * kBN * 2;  // dS^T [128 keys][128 queries] bf16
    static constexpr int kSmemBytes = kOffDS + kBM * kBN * 2 + 1024;
    static constexpr uint32_t kColDK = 0;
    static constexpr uint32_t kColDV = 128;
    static constexpr uint32_t kColST = 256;  // S^T, later dQ
    static constexpr uint32_t kColDP = 384;  // dP^T
    static constexpr uint32_t kTmemCols = 512;
};

struct BwdParams {
    CUtensorMap tm_q;   // local: Q [B,T,Hq,D]; global: packed [1,cap+128,Hq,D]
    CUtensorMap tm_do;  // same layout as tm_q
    CUtensorMap tm_k;   // [B,T,Hkv,D]
    CUtensorMap tm_v;
    const float* lse;   // local [B,Hq,T]; global [Hq,cap]
    const float* dsum;  // same layout as lse
    float* dq_acc;      // local [B,T,Hq,D]; global [cap+128,Hq,D]
    logo_bf16* dk;      // [B,T,Hkv,D]
    logo_bf16* dv;
    const int32_t* pos;
    const int32_t* cu_q;
    const int32_t* first_row;  // global: [B, nblk] first packed row of sequence b whose position reaches block j
    logo_bf16* dq_fill;        // global, d = 128: dense dQ [B, T, Hq, D] whose unselected rows this kernel zeroes
    int B, T, Hq, Hkv, window, cap, nblk, q_tiles;
    float scale, scale_log2;
};

struct BwdItem {
    int b, j, kvh;
    int i_lo, ntiles;   // query tiles visited: i_lo .. i_lo + ntiles - 1
    int row_lo, row_hi; // global: packed rows of sequence b
};

template <bool GLOBAL>
__device__ __forceinline__ BwdItem decode_bwd(const BwdParams& p, int k)
{
    BwdItem it;
    it.kvh = k % p.Hkv;
    const int t = k / p.Hkv;
    it.b = t % p.B;
    it.j = t / p.B;
    const int k0 = it.j * kBN;
    if (!GLOBAL) {
        it.i_lo = it.j;
        const int i_hi = min(p.q_tiles - 1, (k0 + kBN - 1 + p.window - 1) / kBM);
        it.ntiles = i_hi - it.i_lo + 1;
        it.row_lo = it.row_hi = 0;
    } else {
        it.row_lo = p.cu_q[it.b];
        it.row_hi = p.cu_q[it.b + 1];
        // first packed row of the sequence whose position can see key k0
        int lo = it.row_lo, hi = it.row_hi;
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (p.pos[mid] < k0) lo = mid + 1;
            else hi = mid;
        }
        if (lo >= it.row_hi) {
            it.i_lo = 0;
            it.ntiles = 0;
        } else {
            it.i_lo = lo / kBM;
            it.ntiles = (it.row_hi - 1) / kBM - it.i_lo + 1;
        }
    }
    return it;
}

template <int D, bool GLOBAL>
__global__ void __launch_bounds__(192, 1) attn_bwd_kernel(const __grid_constant__ BwdParams p)
{
    using C = BwdCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_kv_full, bar_kv_empty, bar_qdo_full, bar_qdo_empty, bar_st_full,
        bar_ds_full, bar_dq_full, bar_dq_empty, bar_dkv_full, bar_dkv_empty, bar_drain, bar_stage;
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;
    __shared__ int sh_pos[2][kBM];
    __shared__ float sh_lse[2][kBM];
    __shared__ float sh_dsum[2][kBM];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sK = smem_u32(smem + C::kOffK), sV = smem_u32(smem + C::kOffV);
    const uint32_t sQ = smem_u32(smem + C::kOffQ), sDO = smem_u32(smem + C::kOffDO);
    const uint32_t sP = smem_u32(smem + C::kOffP), sDS = smem_u32(smem + C::kOffDS);
    const int group = p.Hq / p.Hkv;
    const int n_items = p.B * p.nblk * p.Hkv;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_kv_full), 1);
        mbar_init(smem_u32(&bar_kv_empty), 1);
        mbar_init(smem_u32(&bar_qdo_full), 1);
        mbar_init(smem_u32(&bar_qdo_empty), 1);
        mbar_init(smem_u32(&bar_st_full), 1);
        mbar_init(smem_u32(&bar_ds_full), 128);
        mbar_init(smem_u32(&bar_dq_full), 1);
        mbar_init(smem_u32(&bar_dq_empty), 128);
        mbar_init(smem_u32(&bar_dkv_full), 1);
        mbar_init(smem_u32(&bar_dkv_empty), 128);
        mbar_init(smem_u32(&bar_drain), 1);
        mbar_init(smem_u32(&bar_stage), 128);
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_base_sh), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&p.tm_q);
            tma_prefetch_desc(&p.tm_do);
            tma_prefetch_desc(&p.tm_k);
            tma_prefetch_desc(&p.tm_v);
            const uint64_t pol_q = policy_evict_last();
            const uint64_t pol_kv = policy_evict_first();
            int u = 0, kv_items = 0;
            bool ok = true;
            for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
                const BwdItem it = decode_bwd<GLOBAL>(p, k);
                if (it.ntiles == 0) continue;
                if (!(ok = mbar_wait(smem_u32(&bar_kv_empty), (kv_items & 1) ^ 1, &abort_flag))) break;
                const uint32_t kvb = smem_u32(&bar_kv_full);
                mbar_arrive_expect_tx(kvb, 2 * C::kTileBytes);
                for (int s = 0; s < C::kSub; ++s) {
                    tma_load_4d(sK + s * 16384, &p.tm_k, kvb, 64 * s, it.kvh, it.j * kBN, it.b, pol_kv);
                    tma_load_4d(sV + s * 16384, &p.tm_v, kvb, 64 * s, it.kvh, it.j * kBN, it.b, pol_kv);
                }
                ++kv_items;
                const int n_it = group * it.ntiles;
                for (int x = 0; x < n_it; ++x, ++u) {
                    const int h = it.kvh * group + x / it.ntiles;
                    const int i = it.i_lo + x % it.ntiles;
                    if (!(ok = mbar_wait(smem_u32(&bar_qdo_empty), (u & 1) ^ 1, &abort_flag))) break;
                    const uint32_t qb = smem_u32(&bar_qdo_full);
                    mbar_arrive_expect_tx(qb, 2 * C::kTileBytes);
                    const int cb = GLOBAL ? 0 : it.b;
                    for (int s = 0; s < C::kSub; ++s) {
                        tma_load_4d(sQ + s * 16384, &p.tm_q, qb, 64 * s, h, i * kBM, cb, pol_q);
                        tma_load_4d(sDO + s * 16384, &p.tm_do, qb, 64 * s, h, i * kBM, cb, pol_q);
                    }
                }
            }
            if (!ok) {
                if (kv_items > 0) mbar_wait_drain(smem_u32(&bar_kv_full), (kv_items - 1) & 1);
                if (u > 0) mbar_wait_drain(smem_u32(&bar_qdo_full), (u - 1) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBM, kBN, false, false);  // S^T, dP^T
            constexpr uint32_t idKM = idesc_bf16_f32(kBM, D, false, true);    // dV, dK
            constexpr uint32_t idMM = idesc_bf16_f32(kBM, D, true, true);     // dQ
            int u = 0, kv_items = 0;
            bool ok = true;
            for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
                const BwdItem it = decode_bwd<GLOBAL>(p, k);
                if (it.ntiles == 0) continue;
                if (!(ok = mbar_wait(smem_u32(&bar_kv_full), kv_items & 1, &abort_flag))) break;
                if (!(ok = mbar_wait(smem_u32(&bar_dkv_empty), (kv_items & 1) ^ 1, &abort_flag))) break;
                const int n_it = group * it.ntiles;
                for (int x = 0; x < n_it; ++x, ++u) {
                    if (!(ok = mbar_wait(smem_u32(&bar_qdo_full), u & 1, &abort_flag))) break;
                    if (!(ok = mbar_wait(smem_u32(&bar_dq_empty), (u & 1) ^ 1, &abort_flag))) break;
                    tc_fence_after();
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks) {
                        const uint32_t off = (ks >> 2) * 16384 + (ks & 3) * 32;
                        umma_bf16_ss(tmem + C::kColST, sdesc_sw128(sK + off, 16, 1024), sdesc_sw128(sQ + off, 16, 1024),
                                     idS, ks > 0 ? 1u : 0u);
                    }
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks) {
                        const uint32_t off = (ks >> 2) * 16384 + (ks & 3) * 32;
                        umma_bf16_ss(tmem + C::kColDP, sdesc_sw128(sV + off, 16, 1024),
                                     sdesc_sw128(sDO + off, 16, 1024), idS, ks > 0 ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_st_full));
                    if (!(ok = mbar_wait(smem_u32(&bar_ds_full), u & 1, &abort_flag))) break;
                    tc_fence_after();
#pragma unroll
                    for (int ks = 0; ks < kBM / 16; ++ks) {
                        const uint32_t koff = (ks >> 2) * 16384 + (ks & 3) * 32;  // K-major step over queries
                        const uint32_t moff = ks * 2048;                           // MN-major step over 16 rows
                        const uint32_t acc = (x > 0 || ks > 0) ? 1u : 0u;
                        umma_bf16_ss(tmem + C::kColDV, sdesc_sw128(sP + koff, 16, 1024),
                                     sdesc_sw128(sDO + moff, 16384, 1024), idKM, acc);
                        umma_bf16_ss(tmem + C::kColDK, sdesc_sw128(sDS + koff, 16, 1024),
                                     sdesc_sw128(sQ + moff, 16384, 1024), idKM, acc);
                    }
#pragma unroll
                    for (int ks = 0; ks < kBN / 16; ++ks) {
                        const uint32_t moff = ks * 2048;  // 16 keys per step
                        umma_bf16_ss(tmem + C::kColST, sdesc_sw128(sDS + moff, 16384, 1024),
                                     sdesc_sw128(sK + moff, 16384, 1024), idMM, ks > 0 ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_dq_full));
                    umma_commit(smem_u32(&bar_qdo_empty));
                }
                if (!ok) break;
                umma_commit(smem_u32(&bar_kv_empty));
                umma_commit(smem_u32(&bar_dkv_full));
                ++kv_items;
            }
            if (!ok) {
                umma_commit(smem_u32(&bar_drain));
                mbar_wait_drain(smem_u32(&bar_drain), 0);
            }
        }
    } else {
        // ------------------------------------------------------------ softmax-bwd / epilogues
        const int quad = warp & 3;
        const int t = quad * 32 + lane;  // key row for P^T/dS^T; query row for dQ
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const int window = GLOBAL ? kNoWindow : p.window;
        int u = 0, kv_items = 0;
        bool ok = true;
        for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
            const BwdItem it = decode_bwd<GLOBAL>(p, k);
            const int key = it.j * kBN + t;
            const int64_t kv_off = ((static_cast<int64_t>(it.b) * p.T + key) * p.Hkv + it.kvh) * D;
            if (it.ntiles == 0) {  // no selected row sees this block: dK = dV = 0
                if (key < p.T) {
                    for (int c = 0; c < D; c += 8) {
                        *reinterpret_cast<uint4*>(p.dk + kv_off + c) = make_uint4(0, 0, 0, 0);
                        *reinterpret_cast<uint4*>(p.dv + kv_off + c) = make_uint4(0, 0, 0, 0);
                    }
                }
                continue;
            }
            const int n_it = group * it.ntiles;
            for (int x = 0; x < n_it; ++x, ++u) {
                const int h = it.kvh * group + x / it.ntiles;
                const int i = it.i_lo + x % it.ntiles;
                const int sb = u & 1;
                // stage this query tile's positions, lse (log2 units) and Dsum
                {
                    int pc = -1;
                    float l2 = 0.f, ds = 0.f;
                    if (!GLOBAL) {
                        const int q = i * kBM + t;
                        if (q < p.T) {
                            const int64_t idx = (static_cast<int64_t>(it.b) * p.Hq + h) * p.T + q;
                            pc = q;
                            l2 = p.lse[idx] * kLog2e;
                            ds = p.dsum[idx];
                        }
                    } else {
                        const int row = i * kBM + t;
                        if (row >= it.row_lo && row < it.row_hi) {
                            const int64_t idx = static_cast<int64_t>(h) * p.cap + row;
                            pc = p.pos[row];
                            l2 = p.lse[idx] * kLog2e;
                            ds = p.dsum[idx];
                        }
                    }
                    sh_pos[sb][t] = pc;
                    sh_lse[sb][t] = l2;
                    sh_dsum[sb][t] = ds;
                }
                // the four compute warps sync on a bounded barrier (never an
                // unbounded bar.sync: an aborting warp must not strand others)
                mbar_arrive(smem_u32(&bar_stage));
                ok = mbar_wait(smem_u32(&bar_stage), u & 1, &abort_flag);
                if (!ok) break;
                ok = mbar_wait(smem_u32(&bar_st_full), u & 1, &abort_flag);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
#pragma unroll 1
                for (int cc = 0; cc < kBM / 32; ++cc) {
                    uint32_t sv[32], dpv[32];
                    tmem_ld32(tmem + lane_off + C::kColST + cc * 32, sv);
                    tmem_ld32(tmem + lane_off + C::kColDP + cc * 32, dpv);
                    tmem_wait_ld();
                    uint32_t pk[16], dk2[16];
#pragma unroll
                    for (int e = 0; e < 32; e += 2) {
                        float pe[2], de[2];
#pragma unroll
                        for (int z = 0; z < 2; ++z) {
                            const int c = cc * 32 + e + z;
                            const int pc = sh_pos[sb][c];
                            const bool vis = key_visible(key, pc, window);
                            const float pr =
                                vis ? ex2_approx(fmaf(__uint_as_float(sv[e + z]), p.scale_log2, -sh_lse[sb][c])) : 0.f;
                            pe[z] = pr;
                            de[z] = pr * (__uint_as_float(dpv[e + z]) - sh_dsum[sb][c]);
                        }
                        pk[e / 2] = pack_bf16x2(pe[0], pe[1]);
                        dk2[e / 2] = pack_bf16x2(de[0], de[1]);
                    }
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        const int chunk = cc * 4 + q4;  // 16-byte chunk index along the query axis
                        const uint32_t off = (chunk >> 3) * 16384 + sw128_offset(t, chunk & 7);
                        st_shared_v4(sP + off, pk[4 * q4], pk[4 * q4 + 1], pk[4 * q4 + 2], pk[4 * q4 + 3]);
                        st_shared_v4(sDS + off, dk2[4 * q4], dk2[4 * q4 + 1], dk2[4 * q4 + 2], dk2[4 * q4 + 3]);
                    }
                }
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_ds_full));
                // dQ of query row t for this (tile, block): fp32 atomics
                ok = mbar_wait(smem_u32(&bar_dq_full), u & 1, &abort_flag);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
                uint32_t dq[D];
#pragma unroll
                for (int cc = 0; cc < D / 32; ++cc) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + C::kColST + cc * 32, v);
                    tmem_wait_ld();
#pragma unroll
                    for (int e = 0; e < 32; ++e) dq[cc * 32 + e] = v[e];
                }
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_dq_empty));
                if (sh_pos[sb][t] >= 0) {
                    float* dst;
                    if (GLOBAL) dst = p.dq_acc + (static_cast<int64_t>(i * kBM + t) * p.Hq + h) * D;
                    else dst = p.dq_acc + ((static_cast<int64_t>(it.b) * p.T + i * kBM + t) * p.Hq + h) * D;
#pragma unroll
                    for (int c = 0; c < D; c += 4) {
                        atomicAdd(reinterpret_cast<float4*>(dst + c),
                                  make_float4(__uint_as_float(dq[c]) * p.scale, __uint_as_float(dq[c + 1]) * p.scale,
                                              __uint_as_float(dq[c + 2]) * p.scale,
                                              __uint_as_float(dq[c + 3]) * p.scale));
                    }
                }
            }
            if (!ok) break;
            // ---- epilogue: dK (scaled) and dV of this KV block
            ok = mbar_wait(smem_u32(&bar_dkv_full), kv_items & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
#pragma unroll
            for (int which = 0; which < 2; ++which) {
                const uint32_t col = which == 0 ? C::kColDK : C::kColDV;
                const float mul = which == 0 ? p.scale : 1.0f;
                logo_bf16* dst = (which == 0 ? p.dk : p.dv) + kv_off;
#pragma unroll
                for (int cc = 0; cc < D / 32; ++cc) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + col + cc * 32, v);
                    tmem_wait_ld();
                    if (key < p.T) {
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {
                            uint4 w;
                            w.x = pack_bf16x2(__uint_as_float(v[8 * q4 + 0]) * mul, __uint_as_float(v[8 * q4 + 1]) * mul);
                            w.y = pack_bf16x2(__uint_as_float(v[8 * q4 + 2]) * mul, __uint_as_float(v[8 * q4 + 3]) * mul);
                            w.z = pack_bf16x2(__uint_as_float(v[8 * q4 + 4]) * mul, __uint_as_float(v[8 * q4 + 5]) * mul);
                            w.w = pack_bf16x2(__uint_as_float(v[8 * q4 + 6]) * mul, __uint_as_float(v[8 * q4 + 7]) * mul);
                            *reinterpret_cast<uint4*>(dst + cc * 32 + q4 * 8) = w;
                        }
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&bar_dkv_empty));
            ++kv_items;
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

// ---------------------------------------------------------------- d = 128
// Overlapped variant for D = 128: query tiles of 64 rows.  S^T and dP^T of a
// tile share one TMEM buffer that the softmax warps release as soon as they
// have loaded it, so the MMAs of tile u+1 run while the softmax works on tile
// u.  P^T goes back to TMEM (two buffers; dV reads it as the TMEM operand),
// dS^T to shared memory (two buffers; dK and dQ^T read it), and dQ is produced
// transposed (dQ^T = K^T dS^T, one TMEM lane per head-dim row).  Roles:
//   warp 0       TMA: K/V per item, Q/dO tiles through a 4-deep ring
//   warp 1       MMA issuer A: S^T, dP^T (M=128 keys, N=64 queries)
//   warp 15      MMA issuer B: once P^T/dS^T of a tile are in shared memory,
//                dV += P^T dO, dK += dS^T Q, dQ^T = K^T dS^T
//   warps 2..9   two warpgroups, one per 32-query half of the tile; thread =
//                key row: P^T and dS^T (bf16) from S^T and dP^T
//   warps 10..13 dQ^T out of TMEM (thread = head-dim row), coalesced fp32
//                atomics into the dQ accumulator (one 128-byte row segment per
//                warp instruction); dK/dV epilogue at the end of each item
//   warp 14      global branch: zero rows of the dense dQ for unselected tokens
struct Bwd2Cfg {
    static constexpr int D = 128;
    static constexpr int kBQ = 64;                 // queries per tile
    static constexpr int kStages = 4;              // Q/dO ring depth
    static constexpr int kKVBytes = kBN * D * 2;   // K or V block: 32 KB
    static constexpr int kQBytes = kBQ * D * 2;    // Q or dO tile: 16 KB (two 8 KB halves of d)
    static constexpr int kPBytes = kBN * kBQ * 2;  // dS^T: 16 KB
    static constexpr int kOffK = 0;
    static constexpr int kOffV = kOffK + kKVBytes;
    static constexpr int kOffQ = kOffV + kKVBytes;
    static constexpr int kOffDO = kOffQ + kStages * kQBytes;
    static constexpr int kOffDS = kOffDO + kStages * kQBytes;  // 2 buffers
    static constexpr int kSmemBytes = kOffDS + 2 * kPBytes + 1024;
    static constexpr uint32_t kColDK = 0;
    static constexpr uint32_t kColDV = 128;
    static constexpr uint32_t kColS = 256;    // S^T (64 cols), dP^T at +64
    static constexpr uint32_t kColDQ = 384;   // dQ^T (64 cols)
    static constexpr uint32_t kColP = 448;    // P^T buffer b (bf16 pairs) at 448 + 32b
    static constexpr uint32_t kTmemCols = 512;
    static constexpr int kThreads = 512;
};

template <bool GLOBAL>
__device__ __forceinline__ BwdItem decode_bwd2(const BwdParams& p, int k)
{
    BwdItem it;
    it.kvh = k % p.Hkv;
    const int t = k / p.Hkv;
    it.b = t % p.B;
    it.j = t / p.B;
    const int k0 = it.j * kBN;
    constexpr int BQ = Bwd2Cfg::kBQ;
    if (!GLOBAL) {
        it.i_lo = k0 / BQ;
        const int i_hi = min((p.T + BQ - 1) / BQ - 1, (k0 + kBN - 1 + p.window - 1) / BQ);
        it.ntiles = i_hi - it.i_lo + 1;
        it.row_lo = it.row_hi = 0;
    } else {
        it.row_lo = p.cu_q[it.b];
        it.row_hi = p.cu_q[it.b + 1];
        const int lo = p.first_row[it.b * p.nblk + it.j];  // precomputed search (App. B)
        if (lo >= it.row_hi) {
            it.i_lo = 0;
            it.ntiles = 0;
        } else {
            it.i_lo = lo / BQ;
            it.ntiles = (it.row_hi - 1) / BQ - it.i_lo + 1;
        }
    }
    return it;
}

template <bool GLOBAL>
__global__ void __launch_bounds__(Bwd2Cfg::kThreads, 1) attn_bwd2_kernel(const __grid_constant__ BwdParams p)
{
    using C = Bwd2Cfg;
    constexpr int D = C::D, BQ = C::kBQ, NS = C::kStages;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_kv_full, bar_kv_empty, bar_dkv_full, bar_dkv_empty, bar_drain, bar_stage;
    __shared__ __align__(8) uint64_t bar_drain_b;
    __shared__ __align__(8) uint64_t bar_qdo_full[NS], bar_qdo_empty[NS];
    __shared__ __align__(8) uint64_t bar_st_full, bar_st_empty;
    __shared__ __align__(8) uint64_t bar_ds_full[2], bar_dq_full[2], bar_dq_empty[2];
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;
    __shared__ int sh_pos[2][BQ];
    // per pair of query columns (2c, 2c+1): (-lse_2c, -lse_2c+1, -Dsum_2c, -Dsum_2c+1), lse in log2 units
    __shared__ float4 sh_pair[2][BQ / 2];
    __shared__ int sh_open[2][2];       // per staging warp: every column sees every key of the block

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sK = smem_u32(smem + C::kOffK), sV = smem_u32(smem + C::kOffV);
    const uint32_t sQ = smem_u32(smem + C::kOffQ), sDO = smem_u32(smem + C::kOffDO);
    const uint32_t sDS = smem_u32(smem + C::kOffDS);
    const int group = p.Hq / p.Hkv;
    const int n_items = p.B * p.nblk * p.Hkv;

    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_kv_full), 1);
        mbar_init(smem_u32(&bar_kv_empty), 1);
        mbar_init(smem_u32(&bar_dkv_full), 1);
        mbar_init(smem_u32(&bar_dkv_empty), 128);
        mbar_init(smem_u32(&bar_drain), 1);
        mbar_init(smem_u32(&bar_drain_b), 1);
        mbar_init(smem_u32(&bar_stage), 256);
        for (int s = 0; s < NS; ++s) {
            mbar_init(smem_u32(&bar_qdo_full[s]), 1);
            mbar_init(smem_u32(&bar_qdo_empty[s]), 1);
        }
        mbar_init(smem_u32(&bar_st_full), 1);
        mbar_init(smem_u32(&bar_st_empty), 256);
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_u32(&bar_ds_full[b]), 256);
            mbar_init(smem_u32(&bar_dq_full[b]), 1);
            mbar_init(smem_u32(&bar_dq_empty[b]), 128);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_base_sh), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&p.tm_q);
            tma_prefetch_desc(&p.tm_do);
            tma_prefetch_desc(&p.tm_k);
            tma_prefetch_desc(&p.tm_v);
            const uint64_t pol_q = policy_evict_last();
            const uint64_t pol_kv = policy_evict_first();
            int u = 0, kv_items = 0;
            bool ok = true;
            for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
                const BwdItem it = decode_bwd2<GLOBAL>(p, k);
                if (it.ntiles == 0) continue;
                if (!(ok = mbar_wait(smem_u32(&bar_kv_empty), (kv_items & 1) ^ 1, &abort_flag))) break;
                const uint32_t kvb = smem_u32(&bar_kv_full);
                mbar_arrive_expect_tx(kvb, 2 * C::kKVBytes);
                for (int s = 0; s < 2; ++s) {
                    tma_load_4d(sK + s * 16384, &p.tm_k, kvb, 64 * s, it.kvh, it.j * kBN, it.b, pol_kv);
                    tma_load_4d(sV + s * 16384, &p.tm_v, kvb, 64 * s, it.kvh, it.j * kBN, it.b, pol_kv);
                }
                ++kv_items;
                const int n_it = group * it.ntiles;
                for (int x = 0; x < n_it; ++x, ++u) {
                    const int h = it.kvh * group + x / it.ntiles;
                    const int i = it.i_lo + x % it.ntiles;
                    const int st = u % NS, f = u / NS;
                    if (!(ok = mbar_wait(smem_u32(&bar_qdo_empty[st]), (f & 1) ^ 1, &abort_flag))) break;
                    const uint32_t qb = smem_u32(&bar_qdo_full[st]);
                    mbar_arrive_expect_tx(qb, 2 * C::kQBytes);
                    const int cb = GLOBAL ? 0 : it.b;
                    for (int s = 0; s < 2; ++s) {
                        tma_load_4d(sQ + st * C::kQBytes + s * 8192, &p.tm_q, qb, 64 * s, h, i * BQ, cb, pol_q);
                        tma_load_4d(sDO + st * C::kQBytes + s * 8192, &p.tm_do, qb, 64 * s, h, i * BQ, cb, pol_q);
                    }
                }
            }
            if (!ok) {  // let copies already issued land before the CTA exits
                if (kv_items > 0) mbar_wait_drain(smem_u32(&bar_kv_full), (kv_items - 1) & 1);
                for (int v = u - NS > 0 ? u - NS : 0; v < u; ++v)
                    mbar_wait_drain(smem_u32(&bar_qdo_full[v % NS]), (v / NS) & 1);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer A: S^T, dP^T
        // The tile's second half (dV, dK, dQ^T) comes from warp 15: two issuing
        // threads keep the tensor pipe fed while either waits for its inputs
        // (the issue queue is short, so one thread that stops to wait starves it).
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBN, BQ, false, false);  // S^T, dP^T: 128 x 64
            int u = 0, kv_items = 0;
            bool ok = true;
            for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
                const BwdItem it = decode_bwd2<GLOBAL>(p, k);
                if (it.ntiles == 0) continue;
                if (!(ok = mbar_wait(smem_u32(&bar_kv_full), kv_items & 1, &abort_flag))) break;
                const int n_it = group * it.ntiles;
                for (int x = 0; x < n_it; ++x, ++u) {
                    const int st = u % NS;
                    if (!(ok = mbar_wait(smem_u32(&bar_qdo_full[st]), (u / NS) & 1, &abort_flag))) break;
                    // the softmax warps have loaded S^T, dP^T of tile u-1
                    if (!(ok = mbar_wait(smem_u32(&bar_st_empty), (u & 1) ^ 1, &abort_flag))) break;
                    tc_fence_after();
                    const uint32_t qb = sQ + st * C::kQBytes, ob = sDO + st * C::kQBytes;
                    const uint32_t scol = tmem + C::kColS;
                    // S^T and dP^T k-steps alternate (two accumulators, both
                    // needed before the softmax can start)
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks) {
                        const uint32_t ka = (ks >> 2) * 16384 + (ks & 3) * 32;
                        const uint32_t kb = (ks >> 2) * 8192 + (ks & 3) * 32;
                        umma_bf16_ss(scol, sdesc_sw128(sK + ka, 16, 1024), sdesc_sw128(qb + kb, 16, 1024), idS,
                                     ks > 0 ? 1u : 0u);
                        umma_bf16_ss(scol + 64, sdesc_sw128(sV + ka, 16, 1024), sdesc_sw128(ob + kb, 16, 1024), idS,
                                     ks > 0 ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_st_full));
                }
                if (!ok) break;
                ++kv_items;
            }
            if (!ok) {
                umma_commit(smem_u32(&bar_drain));
                mbar_wait_drain(smem_u32(&bar_drain), 0);
            }
        }
    } else if (warp == 15) {
        // ------------------------------------------------------------ MMA issuer B: dV, dK, dQ^T
        if (lane == 0) {
            constexpr uint32_t idKV = idesc_bf16_f32(kBN, D, false, true);  // dV, dK: 128 x 128
            constexpr uint32_t idQ = idesc_bf16_f32(D, BQ, true, true);     // dQ^T: 128 x 64
            int u = 0, kv_items = 0;
            bool ok = true;
            for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
                const BwdItem it = decode_bwd2<GLOBAL>(p, k);
                if (it.ntiles == 0) continue;
                const int n_it = group * it.ntiles;
                for (int x = 0; x < n_it; ++x, ++u) {
                    const int b = u & 1, st = u % NS;
                    if (!(ok = mbar_wait(smem_u32(&bar_ds_full[b]), (u >> 1) & 1, &abort_flag))) break;
                    if (x == 0 && !(ok = mbar_wait(smem_u32(&bar_dkv_empty), (kv_items & 1) ^ 1, &abort_flag))) break;
                    tc_fence_after();
                    const uint32_t db = sDS + b * C::kPBytes;
                    const uint32_t qb = sQ + st * C::kQBytes, ob = sDO + st * C::kQBytes;
#pragma unroll
                    for (int ks = 0; ks < BQ / 16; ++ks) {
                        const uint32_t acc = (x > 0 || ks > 0) ? 1u : 0u;
                        umma_bf16_ts(tmem + C::kColDV, tmem + C::kColP + 32 * b + 8 * ks,
                                     sdesc_sw128(ob + ks * 2048, 8192, 1024), idKV, acc);
                        umma_bf16_ss(tmem + C::kColDK, sdesc_sw128(db + ks * 32, 16, 1024),
                                     sdesc_sw128(qb + ks * 2048, 8192, 1024), idKV, acc);
                    }
                    // Q, dO of tile u are read: release the ring stage before dQ^T
                    // (which reads K and dS^T only), so the next load starts earlier
                    umma_commit(smem_u32(&bar_qdo_empty[st]));
                    // dQ^T: the drain warps have read tile u-1's.  Waited for only
                    // now, so that dV and dK never queue behind the drain.
                    if (u > 0 && !(ok = mbar_wait(smem_u32(&bar_dq_empty[b ^ 1]), ((u - 1) >> 1) & 1, &abort_flag)))
                        break;
                    tc_fence_after();
#pragma unroll
                    for (int ks = 0; ks < kBN / 16; ++ks) {
                        umma_bf16_ss(tmem + C::kColDQ, sdesc_sw128(sK + ks * 2048, 16384, 1024),
                                     sdesc_sw128(db + ks * 2048, 16384, 1024), idQ, ks > 0 ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_dq_full[b]));
                }
                if (!ok) break;
                // the item's last reads of K and V (S^T, dP^T of issuer A finished before ds_full)
                umma_commit(smem_u32(&bar_kv_empty));
                umma_commit(smem_u32(&bar_dkv_full));
                ++kv_items;
            }
            if (!ok) {
                umma_commit(smem_u32(&bar_drain_b));
                mbar_wait_drain(smem_u32(&bar_drain_b), 0);
            }
        }
    } else if (warp < 10) {
        // ------------------------------------------------------------ P^T, dS^T
        const int quad = warp & 3;
        const int half = (warp - 2) >> 2;   // query columns half*32 .. half*32+31
        const int t = quad * 32 + lane;     // key row of the block
        const int tw = threadIdx.x - 64;    // 0..255 across both warpgroups
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const int window = GLOBAL ? kNoWindow : p.window;
        int u = 0;
        bool ok = true;
        for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
            const BwdItem it = decode_bwd2<GLOBAL>(p, k);
            if (it.ntiles == 0) continue;
            const int k0 = it.j * kBN;
            const int key = k0 + t;
            const int n_it = group * it.ntiles;
            // staging values of tile x (query position, lse, Dsum; -1 / 0 / 0
            // outside the tile's rows): loaded one tile ahead and used only at
            // the next tile, so no instruction waits for the loads while the
            // current tile is computed
            int pf_pos = -1;
            float pf_lse = 0.f, pf_dsum = 0.f;
            auto load_stage = [&](int x) {
                const int h = it.kvh * group + x / it.ntiles;
                const int i = it.i_lo + x % it.ntiles;
                pf_pos = -1;
                pf_lse = pf_dsum = 0.f;
                if (!GLOBAL) {
                    const int q = i * BQ + tw;
                    if (q < p.T) {
                        const int64_t idx = (static_cast<int64_t>(it.b) * p.Hq + h) * p.T + q;
                        pf_pos = q;
                        pf_lse = p.lse[idx];
                        pf_dsum = p.dsum[idx];
                    }
                } else {
                    const int row = i * BQ + tw;
                    if (row >= it.row_lo && row < it.row_hi) {
                        const int64_t idx = static_cast<int64_t>(h) * p.cap + row;
                        pf_pos = p.pos[row];
                        pf_lse = p.lse[idx];
                        pf_dsum = p.dsum[idx];
                    }
                }
            };
            if (tw < BQ) load_stage(0);
            for (int x = 0; x < n_it; ++x, ++u) {
                const int b = u & 1;
                if (tw < BQ) {
                    // lse in log2 units; "sees every key of the block"
                    const bool pf_open = pf_pos >= k0 + kBN - 1 && (GLOBAL || pf_pos - k0 < window);
                    sh_pos[b][tw] = pf_pos;
                    float* pr = reinterpret_cast<float*>(&sh_pair[b][tw >> 1]);
                    pr[tw & 1] = -(pf_lse * kLog2e);
                    pr[2 + (tw & 1)] = -pf_dsum;
                    const bool all_open = __all_sync(0xffffffffu, pf_open);
                    if (lane == 0) sh_open[b][tw >> 5] = all_open ? 1 : 0;
                }
                mbar_arrive(smem_u32(&bar_stage));
                ok = mbar_wait(smem_u32(&bar_stage), u & 1, &abort_flag);
                if (!ok) break;
                if (tw < BQ && x + 1 < n_it) load_stage(x + 1);
                const bool open = sh_open[b][0] && sh_open[b][1];
                ok = mbar_wait(smem_u32(&bar_st_full), u & 1, &abort_flag);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
                uint32_t sv[32], dpv[32];
                tmem_ld32(tmem + lane_off + C::kColS + half * 32, sv);
                tmem_ld32(tmem + lane_off + C::kColS + 64 + half * 32, dpv);
                tmem_wait_ld();
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_st_empty));  // S^T, dP^T of tile u+1 may now be written
                uint32_t pk[16], dk2[16];
                // P = 2^(S*scale*log2e - lse), dS = P (dP - Dsum), two columns per
                // f32x2 instruction.  Two branch-free copies of the loop (open
                // tiles skip the visibility test) so that the iterations overlap.
                const uint64_t scale2 = f2_pack(p.scale_log2, p.scale_log2);
                auto columns = [&](auto masked) {
                    constexpr bool kMasked = decltype(masked)::value;
#pragma unroll
                    for (int e = 0; e < 32; e += 2) {
                        const int c = half * 32 + e;
                        const float4 q = sh_pair[b][c >> 1];
                        float x0, x1;
                        f2_unpack(f2_fma(f2_pack(__uint_as_float(sv[e]), __uint_as_float(sv[e + 1])), scale2,
                                         f2_pack(q.x, q.y)),
                                  x0, x1);
                        float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
                        if constexpr (kMasked) {
                            p0 = key_visible(key, sh_pos[b][c], window) ? p0 : 0.f;
                            p1 = key_visible(key, sh_pos[b][c + 1], window) ? p1 : 0.f;
                        }
                        const uint64_t pp = f2_pack(p0, p1);
                        const uint64_t t2 =
                            f2_add(f2_pack(__uint_as_float(dpv[e]), __uint_as_float(dpv[e + 1])), f2_pack(q.z, q.w));
                        float d0, d1;
                        f2_unpack(f2_mul(pp, t2), d0, d1);
                        pk[e / 2] = cvt_bf16x2(p0, p1);
                        dk2[e / 2] = cvt_bf16x2(d0, d1);
                    }
                };
                if (open) columns(std::false_type{});
                else columns(std::true_type{});
                // P^T (TMEM) / dS^T (shared) buffer b is free once the MMAs of tile
                // u-2 are done.  Waiting here rather than before the loads lets
                // S^T, dP^T of tile u+1 enter the MMA queue earlier.
                ok = mbar_wait(smem_u32(&bar_dq_full[b]), ((u >> 1) & 1) ^ 1, &abort_flag);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
                // P^T row t: query columns half*32.. as 16 bf16 pairs, the TMEM
                // operand layout (column c holds queries 2c, 2c+1)
                tmem_st16(tmem + lane_off + C::kColP + 32 * b + half * 16, pk);
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const uint32_t off = sw128_offset(t, half * 4 + q4);
                    st_shared_v4(sDS + b * C::kPBytes + off, dk2[4 * q4], dk2[4 * q4 + 1], dk2[4 * q4 + 2],
                                 dk2[4 * q4 + 3]);
                }
                tmem_wait_st();
                fence_proxy_async_smem();
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_ds_full[b]));
            }
        }
    } else if (warp < 14) {
        // ------------------------------------------------------------ dQ drain, dK/dV epilogue
        const int quad = warp & 3;
        const int t = quad * 32 + lane;  // head-dim row of dQ^T; key row of dK/dV
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        int u = 0, kv_items = 0;
        bool ok = true;
        for (int k = blockIdx.x; k < n_items && ok; k += gridDim.x) {
            const BwdItem it = decode_bwd2<GLOBAL>(p, k);
            const int key = it.j * kBN + t;
            const int64_t kv_off = ((static_cast<int64_t>(it.b) * p.T + key) * p.Hkv + it.kvh) * D;
            if (it.ntiles == 0) {
                // no selected query sees the block: zero dK, dV rows, two whole
                // rows (16 lanes x 16 bytes each) per warp store, this warp's 32 keys
                static_assert(D == 128, "two rows of 16 vectors per warp store");
                for (int r = quad * 32 + (lane >> 4); r < quad * 32 + 32; r += 2) {
                    const int kr = it.j * kBN + r;
                    if (kr < p.T) {
                        const int64_t off =
                            ((static_cast<int64_t>(it.b) * p.T + kr) * p.Hkv + it.kvh) * D + (lane & 15) * 8;
                        *reinterpret_cast<uint4*>(p.dk + off) = make_uint4(0, 0, 0, 0);
                        *reinterpret_cast<uint4*>(p.dv + off) = make_uint4(0, 0, 0, 0);
                    }
                }
                continue;
            }
            const int n_it = group * it.ntiles;
            for (int x = 0; x < n_it; ++x, ++u) {
                const int h = it.kvh * group + x / it.ntiles;
                const int i = it.i_lo + x % it.ntiles;
                const int b = u & 1;
                ok = mbar_wait(smem_u32(&bar_dq_full[b]), (u >> 1) & 1, &abort_flag);
                __syncwarp();
                if (!ok) break;
                tc_fence_after();
                uint32_t v0[32], v1[32];
                tmem_ld32(tmem + lane_off + C::kColDQ, v0);
                tmem_ld32(tmem + lane_off + C::kColDQ + 32, v1);
                tmem_wait_ld();
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_dq_empty[b]));
                // column c of dQ^T is query row c of the tile: rows outside the
                // tile's valid range carry exact zeros (dS = 0 there) and land in
                // padded or neighbouring accumulator rows
                float* base;
                if (GLOBAL) base = p.dq_acc + static_cast<int64_t>(i * BQ) * p.Hq * D + h * D + t;
                else base = p.dq_acc + (static_cast<int64_t>(it.b) * p.T + i * BQ) * p.Hq * D + h * D + t;
                const int64_t rs = static_cast<int64_t>(p.Hq) * D;
#pragma unroll
                for (int c = 0; c < 32; ++c) atomicAdd(base + c * rs, __uint_as_float(v0[c]) * p.scale);
#pragma unroll
                for (int c = 0; c < 32; ++c) atomicAdd(base + (32 + c) * rs, __uint_as_float(v1[c]) * p.scale);
            }
            if (!ok) break;
            ok = mbar_wait(smem_u32(&bar_dkv_full), kv_items & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
#pragma unroll
            for (int which = 0; which < 2; ++which) {
                const uint32_t col = which == 0 ? C::kColDK : C::kColDV;
                const float mul = which == 0 ? p.scale : 1.0f;
                logo_bf16* dst = (which == 0 ? p.dk : p.dv) + kv_off;
#pragma unroll
                for (int cc = 0; cc < D / 32; ++cc) {
                    uint32_t v[32];
                    tmem_ld32(tmem + lane_off + col + cc * 32, v);
                    tmem_wait_ld();
                    if (key < p.T) {
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {
                            uint4 w;
                            w.x = pack_bf16x2(__uint_as_float(v[8 * q4 + 0]) * mul, __uint_as_float(v[8 * q4 + 1]) * mul);
                            w.y = pack_bf16x2(__uint_as_float(v[8 * q4 + 2]) * mul, __uint_as_float(v[8 * q4 + 3]) * mul);
                            w.z = pack_bf16x2(__uint_as_float(v[8 * q4 + 4]) * mul, __uint_as_float(v[8 * q4 + 5]) * mul);
                            w.w = pack_bf16x2(__uint_as_float(v[8 * q4 + 6]) * mul, __uint_as_float(v[8 * q4 + 7]) * mul);
                            *reinterpret_cast<uint4*>(dst + cc * 32 + q4 * 8) = w;
                        }
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(smem_u32(&bar_dkv_empty));
            ++kv_items;
        }
    } else if (GLOBAL && p.dq_fill) {
        // ------------------------------------------------------------ dQ zero fill
        // warp 14: zero the dense dQ rows of the tokens that were not selected
        // (the conversion after this kernel writes only the selected rows).  This
        // kernel leaves nearly all of HBM's bandwidth idle; a separate pass
        // writing the whole dense tensor would not.
        const int64_t ntok = static_cast<int64_t>(p.B) * p.T;
        const int64_t per = (ntok + gridDim.x - 1) / gridDim.x;
        const int64_t t_begin = static_cast<int64_t>(blockIdx.x) * per;
        const int64_t t_end = t_begin + per < ntok ? t_begin + per : ntok;
        const int row_vecs = p.Hq * D / 8;  // 16-byte vectors per token row
        int cur_b = -1, r = 0, r_hi = 0;
        for (int64_t bt = t_begin; bt < t_end; ++bt) {
            const int b = static_cast<int>(bt / p.T), t = static_cast<int>(bt % p.T);
            if (b != cur_b) {  // first packed row of sequence b at or after position t
                cur_b = b;
                int lo = p.cu_q[b], hi = p.cu_q[b + 1];
                r_hi = hi;
                while (lo < hi) {
                    const int mid = (lo + hi) >> 1;
                    if (p.pos[mid] < t) lo = mid + 1;
                    else hi = mid;
                }
                r = lo;
            }
            if (r < r_hi && p.pos[r] == t) {  // selected: converted later
                ++r;
                continue;
            }
            uint4* dst = reinterpret_cast<uint4*>(p.dq_fill + bt * p.Hq * D);
            for (int v = lane; v < row_vecs; v += 32) dst[v] = make_uint4(0u, 0u, 0u, 0u);
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

// ---------------------------------------------------------------- pre / post
// Per (row, head): Dsum = sum_d dO * O (fp32); zero the dQ accumulator rows.
// Global branch: also copy dO_c into the workspace and gather the selected
// rows of the dense Q into the packed layout (App. B), zero-padding the 128
// rows after the last selected one so that partial tiles read finite values;
// and build, for every sequence b and KV block j, the first packed row of b
// whose position reaches the block's first key (App. B's precomputed search
// that lets the backward skip every query tile before it).
struct GlobalPrep {
    const logo_bf16* q;   // dense [B, T, H, D]
    const int32_t* pos;
    const int32_t* cu_q;
    logo_bf16* qc;        // packed [cap + 128, H, D]
    int32_t* first_row;   // [B, nblk]
    int B, nblk;
};

template <bool GLOBAL>
__global__ void __launch_bounds__(128) bwd_pre_kernel(const logo_bf16* __restrict__ o, const logo_bf16* __restrict__ dO,
                                                      const int32_t* __restrict__ n_sel, int rows_host, int T, int H,
                                                      int D, int cap, float* __restrict__ dsum,
                                                      logo_bf16* __restrict__ do_copy, float* __restrict__ dq_acc,
                                                      GlobalPrep gp)
{
    const int n = GLOBAL ? *n_sel : rows_host;
    const int rows = GLOBAL ? n + kBM : rows_host;
    const int vpr = D / 8, nvec = H * vpr;
    if (GLOBAL) {
        for (int idx = blockIdx.x * blockDim.x + threadIdx.x; idx < gp.B * gp.nblk; idx += gridDim.x * blockDim.x) {
            const int b = idx / gp.nblk, j = idx % gp.nblk;
            int lo = gp.cu_q[b], hi = gp.cu_q[b + 1];
            const int k0 = j * kBN;
            while (lo < hi) {
                const int mid = (lo + hi) >> 1;
                if (gp.pos[mid] < k0) lo = mid + 1;
                else hi = mid;
            }
            gp.first_row[idx] = lo;
        }
    }
    for (int row = blockIdx.x; row < rows; row += gridDim.x) {
        const bool live = row < n;
        const int64_t base = static_cast<int64_t>(row) * H * D;
        if (GLOBAL) {
            uint4* dst = reinterpret_cast<uint4*>(gp.qc + base);
            if (live) {
                const int b = seq_of_row(gp.cu_q, gp.B, row);
                const uint4* src = reinterpret_cast<const uint4*>(gp.q + (static_cast<int64_t>(b) * T + gp.pos[row]) * H * D);
                for (int v = threadIdx.x; v < nvec; v += blockDim.x) dst[v] = src[v];
            } else {
                for (int v = threadIdx.x; v < nvec; v += blockDim.x) dst[v] = make_uint4(0, 0, 0, 0);
            }
        }
        for (int v0 = 0; v0 < nvec; v0 += blockDim.x) {
            const int v = v0 + threadIdx.x;
            const bool active = v < nvec;
            const int h = active ? v / vpr : 0, jj = active ? v % vpr : 0;
            float acc = 0.f;
            uint4 graw = make_uint4(0, 0, 0, 0);
            if (active && live) {
                graw = *reinterpret_cast<const uint4*>(dO + base + h * D + jj * 8);
                const uint4 oraw = *reinterpret_cast<const uint4*>(o + base + h * D + jj * 8);
                const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&graw);
                const __nv_bfloat162* o2 = reinterpret_cast<const __nv_bfloat162*>(&oraw);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const float2 a = __bfloat1622float2(g2[e]), b = __bfloat1622float2(o2[e]);
                    acc = fmaf(a.x, b.x, acc);
                    acc = fmaf(a.y, b.y, acc);
                }
            }
            for (int off = vpr >> 1; off > 0; off >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, off);
            if (active) {
                if (GLOBAL) *reinterpret_cast<uint4*>(do_copy + base + h * D + jj * 8) = graw;
                float4* z = reinterpret_cast<float4*>(dq_acc + base + h * D + jj * 8);
                z[0] = make_float4(0.f, 0.f, 0.f, 0.f);
                z[1] = make_float4(0.f, 0.f, 0.f, 0.f);
                if (live && jj == 0) {
                    if (GLOBAL) dsum[static_cast<int64_t>(h) * cap + row] = acc;
                    else {
                        const int b = row / T, tt = row % T;
                        dsum[(static_cast<int64_t>(b) * H + h) * T + tt] = acc;
                    }
                }
            }
        }
    }
}

// Global branch, d = 128: dQ accumulator rows of the selected tokens -> their
// rows of the dense dq (the backward kernel zeroed the others); blocks stride
// over the packed rows below the selected count.
__global__ void __launch_bounds__(128) bwd_post_selected_kernel(const float* __restrict__ dq_acc,
                                                                const int32_t* __restrict__ pos,
                                                                const int32_t* __restrict__ cu_q,
                                                                const int32_t* __restrict__ n_sel, int B, int T, int H,
                                                                int D, logo_bf16* __restrict__ dq)
{
    const int n = *n_sel;
    const int row_elems = H * D;
    for (int r = blockIdx.x; r < n; r += gridDim.x) {
        const int b = seq_of_row(cu_q, B, r);
        const int64_t dst_row = static_cast<int64_t>(b) * T + pos[r];
        for (int v = threadIdx.x; v < row_elems / 8; v += blockDim.x) {
            const float4* s = reinterpret_cast<const float4*>(dq_acc + static_cast<int64_t>(r) * row_elems + v * 8);
            const float4 a = s[0], c = s[1];
            uint4 w;
            w.x = pack_bf16x2(a.x, a.y);
            w.y = pack_bf16x2(a.z, a.w);
            w.z = pack_bf16x2(c.x, c.y);
            w.w = pack_bf16x2(c.z, c.w);
            *reinterpret_cast<uint4*>(dq + dst_row * row_elems + v * 8) = w;
        }
    }
}

// dQ accumulator (fp32) -> dq (bf16).  Local: elementwise.  Global: every
// dense token writes its packed row's gradient, or zeros if not selected.
template <bool GLOBAL>
__global__ void __launch_bounds__(128) bwd_post_kernel(const float* __restrict__ dq_acc, const int32_t* __restrict__ pos,
                                                       const int32_t* __restrict__ cu_q, int T, int H, int D,
                                                       logo_bf16* __restrict__ dq)
{
    const int64_t bt = blockIdx.x;
    const int row_elems = H * D;
    int64_t src_row = bt;
    if (GLOBAL) {
        const int b = static_cast<int>(bt / T), t = static_cast<int>(bt % T);
        int lo = cu_q[b], hi = cu_q[b + 1];
        while (lo < hi) {
            const int mid = (lo + hi) >> 1;
            if (pos[mid] < t) lo = mid + 1;
            else hi = mid;
        }
        src_row = (lo < cu_q[b + 1] && pos[lo] == t) ? lo : -1;
    }
    for (int v = threadIdx.x; v < row_elems / 8; v += blockDim.x) {
        uint4 w = make_uint4(0, 0, 0, 0);
        if (src_row >= 0) {
            const float4* s = reinterpret_cast<const float4*>(dq_acc + src_row * row_elems + v * 8);
            const float4 a = s[0], c = s[1];
            w.x = pack_bf16x2(a.x, a.y);
            w.y = pack_bf16x2(a.z, a.w);
            w.z = pack_bf16x2(c.x, c.y);
            w.w = pack_bf16x2(c.z, c.w);
        }
        *reinterpret_cast<uint4*>(dq + bt * row_elems + v * 8) = w;
    }
}

struct BwdWs {
    logo_bf16* qc;
    logo_bf16* doc;
    float* dsum;
    float* dq_acc;
    int32_t* first_row;
};

size_t local_bwd_ws_layout(const logo_dims& d, char* base, BwdWs* ws)
{
    const size_t rows = static_cast<size_t>(d.B) * d.T;
    size_t off = 0;
    const size_t o_ds = off;
    off = round_up(off + rows * d.Hq * sizeof(float), 256);
    const size_t o_dq = off;
    off = round_up(off + (rows + kBM) * d.Hq * d.D * sizeof(float), 256);
    if (ws) {
        ws->qc = ws->doc = nullptr;
        ws->dsum = reinterpret_cast<float*>(base + o_ds);
        ws->dq_acc = reinterpret_cast<float*>(base + o_dq);
        ws->first_row = nullptr;
    }
    return off;
}

size_t global_bwd_ws_layout(const logo_dims& d, char* base, BwdWs* ws)
{
    const size_t cap = static_cast<size_t>(d.B) * d.T;
    const size_t rows = cap + kBM;
    size_t off = 0;
    const size_t o_qc = off;
    off = round_up(off + rows * d.Hq * d.D * 2, 256);
    const size_t o_do = off;
    off = round_up(off + rows * d.Hq * d.D * 2, 256);
    const size_t o_ds = off;
    off = round_up(off + cap * d.Hq * sizeof(float), 256);
    const size_t o_dq = off;
    off = round_up(off + rows * d.Hq * d.D * sizeof(float), 256);
    const size_t o_fr = off;
    off = round_up(off + static_cast<size_t>(d.B) * ((d.T + kBN - 1) / kBN) * sizeof(int32_t), 256);
    if (ws) {
        ws->first_row = reinterpret_cast<int32_t*>(base + o_fr);
        ws->qc = reinterpret_cast<logo_bf16*>(base + o_qc);
        ws->doc = reinterpret_cast<logo_bf16*>(base + o_do);
        ws->dsum = reinterpret_cast<float*>(base + o_ds);
        ws->dq_acc = reinterpret_cast<float*>(base + o_dq);
    }
    return off;
}

template <int D, bool GLOBAL>
int launch_bwd(const BwdParams& prm, cudaStream_t st)
{
    static bool attr_done = false;  // benign race: setting the attribute twice is harmless
    const int n_items = prm.B * prm.nblk * prm.Hkv;
    const int grid = max(1, min(n_items, device_sm_count()));
    if (D == 128) {
        if (!attr_done) {
            if (set_smem_limit(attn_bwd2_kernel<GLOBAL>, Bwd2Cfg::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
            attr_done = true;
        }
        attn_bwd2_kernel<GLOBAL><<<grid, Bwd2Cfg::kThreads, Bwd2Cfg::kSmemBytes, st>>>(prm);
    } else {
        using C = BwdCfg<D>;
        if (!attr_done) {
            if (set_smem_limit(attn_bwd_kernel<D, GLOBAL>, C::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
            attr_done = true;
        }
        attn_bwd_kernel<D, GLOBAL><<<grid, 192, C::kSmemBytes, st>>>(prm);
    }
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

int check_bwd_ptrs(const void* const* ptrs, int n)
{
    for (int i = 0; i < n; ++i) {
        if (!ptrs[i]) return LOGO_ERR_INVALID_ARG;
        if (!aligned16(ptrs[i])) return LOGO_ERR_UNSUPPORTED;
    }
    return LOGO_OK;
}

}  // namespace

int attn_bwd_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" size_t logo_local_attn_bwd_workspace_size(logo_dims dims)
{
    if (check_dims(dims) != LOGO_OK) return 0;
    return local_bwd_ws_layout(dims, nullptr, nullptr);
}

extern "C" int logo_local_attn_bwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, const logo_bf16* o,
                                   const float* lse, const logo_bf16* dO, logo_bf16* dq, logo_bf16* dk,
                                   logo_bf16* dv, logo_dims dims, int window, float scale, void* workspace,
                                   size_t workspace_bytes, void* stream)
{
    int rc = check_dims(dims);
    if (rc != LOGO_OK) return rc;
    const void* ptrs[] = {q, k, v, o, dO, dq, dk, dv};
    if ((rc = check_bwd_ptrs(ptrs, 8)) != LOGO_OK) return rc;
    if (!lse || window < 1) return LOGO_ERR_INVALID_ARG;
    if (!(scale >= 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (scale == 0.0f) scale = 1.0f / sqrtf(static_cast<float>(dims.D));
    const size_t need = local_bwd_ws_layout(dims, nullptr, nullptr);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return LOGO_ERR_WORKSPACE;
    BwdWs ws;
    local_bwd_ws_layout(dims, static_cast<char*>(workspace), &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int rows = dims.B * dims.T;
    const int pre_grid = max(1, min(rows, device_sm_count() * 16));
    bwd_pre_kernel<false><<<pre_grid, 128, 0, st>>>(o, dO, nullptr, rows, dims.T, dims.Hq, dims.D, 0, ws.dsum,
                                                    nullptr, ws.dq_acc, GlobalPrep{});
    BwdParams prm{};
    const uint32_t qrows = dims.D == 128 ? Bwd2Cfg::kBQ : kBM;
    if (!encode_bf16_4d(&prm.tm_q, q, dims.D, dims.Hq, dims.T, dims.B, 64, qrows) ||
        !encode_bf16_4d(&prm.tm_do, dO, dims.D, dims.Hq, dims.T, dims.B, 64, qrows) ||
        !encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN))
        return LOGO_ERR_CUDA;
    prm.lse = lse;
    prm.dsum = ws.dsum;
    prm.dq_acc = ws.dq_acc;
    prm.dk = dk;
    prm.dv = dv;
    prm.B = dims.B;
    prm.T = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = window > dims.T ? dims.T : window;
    prm.cap = rows;
    prm.nblk = (dims.T + kBN - 1) / kBN;
    prm.q_tiles = (dims.T + kBM - 1) / kBM;
    prm.scale = scale;
    prm.scale_log2 = scale * kLog2e;
    rc = dims.D == 128 ? launch_bwd<128, false>(prm, st) : launch_bwd<64, false>(prm, st);
    if (rc != LOGO_OK) return rc;
    bwd_post_kernel<false><<<rows, 128, 0, st>>>(ws.dq_acc, nullptr, nullptr, dims.T, dims.Hq, dims.D, dq);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

extern "C" size_t logo_global_attn_bwd_workspace_size(logo_dims dims)
{
    if (check_dims(dims) != LOGO_OK) return 0;
    return global_bwd_ws_layout(dims, nullptr, nullptr);
}

extern "C" int logo_global_sparse_attn_bwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v,
                                           const int32_t* pos, const int32_t* cu_q, const int32_t* n_sel_total,
                                           const logo_bf16* o_c, const float* lse_c, const logo_bf16* dO_c,
                                           logo_bf16* dq, logo_bf16* dk, logo_bf16* dv, logo_dims dims, float scale,
                                           void* workspace, size_t workspace_bytes, void* stream)
{
    int rc = check_dims(dims);
    if (rc != LOGO_OK) return rc;
    const void* ptrs[] = {q, k, v, o_c, dO_c, dq, dk, dv};
    if ((rc = check_bwd_ptrs(ptrs, 8)) != LOGO_OK) return rc;
    if (!pos || !cu_q || !n_sel_total || !lse_c) return LOGO_ERR_INVALID_ARG;
    if (!(scale >= 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (scale == 0.0f) scale = 1.0f / sqrtf(static_cast<float>(dims.D));
    const size_t need = global_bwd_ws_layout(dims, nullptr, nullptr);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return LOGO_ERR_WORKSPACE;
    BwdWs ws;
    global_bwd_ws_layout(dims, static_cast<char*>(workspace), &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int cap = dims.B * dims.T;
    const int grid_rows = max(1, min(cap + kBM, device_sm_count() * 16));
    const int nblk = (dims.T + kBN - 1) / kBN;
    const GlobalPrep gp{q, pos, cu_q, ws.qc, ws.first_row, dims.B, nblk};
    bwd_pre_kernel<true><<<grid_rows, 128, 0, st>>>(o_c, dO_c, n_sel_total, 0, dims.T, dims.Hq, dims.D, cap, ws.dsum,
                                                    ws.doc, ws.dq_acc, gp);
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    BwdParams prm{};
    const uint32_t qrows = dims.D == 128 ? Bwd2Cfg::kBQ : kBM;
    if (!encode_bf16_4d(&prm.tm_q, ws.qc, dims.D, dims.Hq, static_cast<uint64_t>(cap) + kBM, 1, 64, qrows) ||
        !encode_bf16_4d(&prm.tm_do, ws.doc, dims.D, dims.Hq, static_cast<uint64_t>(cap) + kBM, 1, 64, qrows) ||
        !encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN))
        return LOGO_ERR_CUDA;
    prm.lse = lse_c;
    prm.dsum = ws.dsum;
    prm.dq_acc = ws.dq_acc;
    prm.dk = dk;
    prm.dv = dv;
    prm.pos = pos;
    prm.cu_q = cu_q;
    prm.first_row = ws.first_row;
    prm.dq_fill = dims.D == 128 ? dq : nullptr;
    prm.B = dims.B;
    prm.T = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = kNoWindow;
    prm.cap = cap;
    prm.nblk = (dims.T + kBN - 1) / kBN;
    prm.q_tiles = 0;
    prm.scale = scale;
    prm.scale_log2 = scale * kLog2e;
    rc = dims.D == 128 ? launch_bwd<128, true>(prm, st) : launch_bwd<64, true>(prm, st);
    if (rc != LOGO_OK) return rc;
    if (dims.D == 128)
        bwd_post_selected_kernel<<<grid_rows, 128, 0, st>>>(ws.dq_acc, pos, cu_q, n_sel_total, dims.B, dims.T,
                                                            dims.Hq, dims.D, dq);
    else
        bwd_post_kernel<true><<<cap, 128, 0, st>>>(ws.dq_acc, pos, cu_q, dims.T, dims.Hq, dims.D, dq);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
