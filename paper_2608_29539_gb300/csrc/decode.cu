// decode.cu -- one decoding step of both attention branches, compacting the
// global branch to the selected sequences (Sec. 3.3 Autoregressive Decoding:
// the gate is known before the global call, so unselected tokens skip it; the
// paper's serving path launches a dense call and masks, and leaves a kernel
// that compacts active decode rows as the missing piece).
//
//   logo_decode_local_attn          every sequence's new token attends the last
//                                   W positions, read from a ring cache (Eq. 6)
//   logo_decode_global_sparse_attn  only the packed selected rows attend their
//                                   sequence's whole dense cache (Eq. 8)
//
// Both run one persistent kernel per call.  An item is one chunk of cache
// rows (up to kDecSubMax sub-tiles of 64 rows) of one (row, KV head); a CTA
// (4 warps) walks its items' sub-tiles through a 3-stage TMA ring (128-byte
// swizzle), a stage refilled once all four warps have released it, and
// serves every query head of the KV head's group from each: S = q.K^T and
// O = P.V as warp-level bf16 products (mma.sync m16n8k16: the group's heads
// are the 16 rows, so a group of up to 16 heads fills one tile).  Each warp
// takes 16 rows of every sub-tile and keeps its own online softmax (running
// max and sum per head, in log2 units) across the item's sub-tiles, P going
// from the S fragments straight into the A fragments of the P.V product, so
// nothing inside the sub-tile loop waits for another warp; the four warps'
// results are combined exactly at the end of the item.
// A row whose cache fits one chunk gets its output written by that item.
// Longer caches are split into chunks for parallelism: each chunk leaves its
// unnormalised O, max and sum, and the last chunk of a (row, KV head) to
// finish (a counter per pair, cleared by the call) combines them exactly.
// Decoding is bound by HBM: every cache byte serves only the group's heads.
// In the global call the items of rows past the device-side count of
// selected rows are never visited, so unselected sequences cost no cache
// traffic and no host synchronisation is needed.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>

#include "attn_common.cuh"
#include "host_common.h"
#include "logo_status.cuh"
#include "sm100.cuh"

namespace logo {
namespace {

constexpr int kDecThreads = 128;  // 4 warps
constexpr int kDecRows = 64;      // cache rows per sub-tile, 16 per warp
constexpr int kDecRowsPerWarp = kDecRows / 4;
constexpr int kDecMaxGroup = 16;  // query heads per KV head (the mma tile's 16 rows)
constexpr int kDecSubMax = 16;    // sub-tiles per chunk preferred at most (1024 cache rows): the merge walks a row's chunks serially
constexpr int kDecStages = 3;     // TMA ring depth

struct DecParams {
    CUtensorMap tm_k;  // cache [B, R, Hkv, D], box {64, 1, 128, 1}
    CUtensorMap tm_v;
    const logo_bf16* q;       // [B, Hq, D]
    const int32_t* seq_len;   // [B] tokens in the cache, the new one included
    const int32_t* cu_q;      // global: [B+1] packed rows of the (B, 1) selection
    const int32_t* n_sel;     // global: [1]
    float* part;              // [rows, Hq, nchunk, D + 2]: unnormalised o, then m, l (nchunk > 1)
    int32_t* done;            // [rows, Hkv] chunks finished (nchunk > 1; cleared by the call)
    logo_bf16* out;           // [B, Hq, D] (global: packed rows)
    int B, R, Hq, Hkv, window, nchunk, sub_per_chunk;
    float scale_log2;
};

template <int D>
struct DecCfg {
    static constexpr int kHalfBytes = kDecRows * 128;         // 64 head-dim columns of the sub-tile's rows
    static constexpr int kTileBytes = (D / 64) * kHalfBytes;  // K or V sub-tile
    static constexpr int kStageBytes = 2 * kTileBytes;        // K then V
    static constexpr int kOffW = kDecStages * kStageBytes;    // chunk-merge weights [group][chunks] fp32
    static constexpr int kOffM = kOffW + 16 * 64 * 4;         // the warps' partial results, sized per group:
    // [warp][group][D + 2] fp32: unnormalised o, then m, l
    static constexpr int merge_bytes(int group) { return 4 * group * (D + 2) * 4; }
    static constexpr int smem_bytes(int group) { return kOffM + merge_bytes(group) + 1024; }
};
constexpr int kDecMaxChunks = 64;  // chunks per cache at most (the merge's weights: group x chunks <= 16 x 64)

// Row j of the cache holds position pos_of(j) (or none: -1).  Dense cache:
// j itself while j < len.  Ring of R slots: the latest position congruent to j
// modulo R that is in the cache.
template <bool RING>
__device__ __forceinline__ int pos_of(int j, int len, int R)
{
    if (j >= len) return -1;
    return RING ? j + R * ((len - 1 - j) / R) : j;
}

// One item's place in the call: row r (sequence b), KV head, chunk c; its
// sub-tiles [s0, s1) of the cache (empty when the chunk lies past the rows used).
struct DecItem {
    int r, b, kvh, c, len, s0, s1, nused;  // nused: chunks of the row holding cache rows
};

template <bool RING>
__device__ __forceinline__ DecItem dec_item(const DecParams& p, long long w)
{
    DecItem it;
    it.c = static_cast<int>(w % p.nchunk);
    const long long t = w / p.nchunk;
    it.kvh = static_cast<int>(t % p.Hkv);
    it.r = static_cast<int>(t / p.Hkv);
    it.b = RING ? it.r : seq_of_row(p.cu_q, p.B, it.r);
    it.len = RING ? p.seq_len[it.b] : min(p.seq_len[it.b], p.R);  // a dense cache holds at most R tokens
    const int rows_used = max(0, min(it.len, p.R));
    const int subs = (rows_used + kDecRows - 1) / kDecRows;
    it.nused = (subs + p.sub_per_chunk - 1) / p.sub_per_chunk;
    it.s0 = it.c * p.sub_per_chunk;
    it.s1 = min(subs, it.s0 + p.sub_per_chunk);
    if (it.len < 1 || it.s0 >= it.s1) it.s1 = it.s0;  // nothing to do
    return it;
}

template <int D, bool RING>
__global__ void __launch_bounds__(kDecThreads, 2) decode_attn_kernel(const __grid_constant__ DecParams p)
{
    using C = DecCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    // bar_full: a stage's K/V sub-tile landed; bar_empty: the four warps are done with it
    __shared__ __align__(8) uint64_t bar_full[kDecStages], bar_empty[kDecStages];
    __shared__ volatile int abort_flag;
    __shared__ int sh_last;
    __shared__ float sh_wm[4][kDecMaxGroup];  // per head: weight of each warp's partial, 1 / L
    __shared__ float sh_M[kDecMaxGroup], sh_L[kDecMaxGroup];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gid = lane >> 2, tig = lane & 3;  // mma fragment coordinates
    const int mi = lane >> 3, rr = lane & 7;    // ldmatrix: matrix index, row in the matrix
    const int group = p.Hq / p.Hkv;
    float* sW = reinterpret_cast<float*>(smem + C::kOffW);
    float* sM = reinterpret_cast<float*>(smem + C::kOffM);
    const uint32_t sRing = smem_u32(smem);
    // rows of the call: every sequence (local), the selected packed rows (global)
    const int n_rows = RING ? p.B : *p.n_sel;
    const long long n_items = static_cast<long long>(n_rows) * p.Hkv * p.nchunk;
    if (tid == 0) {
        abort_flag = 0;
        for (int s = 0; s < kDecStages; ++s) {
            mbar_init(smem_u32(&bar_full[s]), 1);
            mbar_init(smem_u32(&bar_empty[s]), 4);
        }
        fence_mbar_init();
    }
    __syncthreads();

    // ---- the producer (thread 0) walks the same sequence of sub-tiles as the
    //      consumers, up to kDecStages ahead: (item w, sub-tile s) in order; a
    //      stage is refilled once every warp has released it
    long long pw = blockIdx.x;
    int ps = 0, ps1 = 0;
    auto producer_next = [&](DecItem* it_out) -> bool {  // the next sub-tile to load, or false
        while (ps >= ps1) {
            if (pw >= n_items) return false;
            const DecItem it = dec_item<RING>(p, pw);
            pw += gridDim.x;
            ps = it.s0;
            ps1 = it.s1;
            *it_out = it;
        }
        return true;
    };
    DecItem pit{};
    int issued = 0;
    bool ok = true;
    auto issue = [&]() {
        if (tid != 0 || !ok) return;
        if (!producer_next(&pit)) return;
        const int st = issued % kDecStages;
        if (!(ok = mbar_wait(smem_u32(&bar_empty[st]), ((issued / kDecStages) & 1) ^ 1, &abort_flag))) return;
        const uint32_t bar = smem_u32(&bar_full[st]);
        const uint32_t base = sRing + st * C::kStageBytes;
        const uint64_t pol = policy_evict_first();
        mbar_arrive_expect_tx(bar, C::kStageBytes);
        for (int h = 0; h < D / 64; ++h) {
            tma_load_4d(base + h * C::kHalfBytes, &p.tm_k, bar, 64 * h, pit.kvh, ps * kDecRows, pit.b, pol);
            tma_load_4d(base + C::kTileBytes + h * C::kHalfBytes, &p.tm_v, bar, 64 * h, pit.kvh, ps * kDecRows, pit.b,
                        pol);
        }
        ++ps;
        ++issued;
    };
    for (int i = 0; i < kDecStages - 1; ++i) issue();

    // Each warp takes 16 rows of every sub-tile (rows 16w..16w+15) and keeps an
    // online softmax of its own across the item's sub-tiles, so no instruction
    // inside the sub-tile loop waits for another warp: S = q.K^T lands in mma
    // fragments, P = 2^(S - m) goes from those straight into the A fragments
    // of O += P.V (a pair of 8-column S tiles is one 16-deep A fragment), and
    // the four warps' results are combined once per item.
    constexpr int NT = D / 8;
    int consumed = 0;
    for (long long w = blockIdx.x; w < n_items && ok; w += gridDim.x) {
        const DecItem it = dec_item<RING>(p, w);
        if (it.s0 >= it.s1) continue;
        const int h0 = it.kvh * group;
        // the group's queries as mma A fragments (rows = heads, zero past the group)
        uint32_t qa[D / 16][4];
        {
            const logo_bf16* q0 = p.q + (static_cast<int64_t>(it.b) * p.Hq + h0) * D;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int hh = gid + (i & 1) * 8;
                    const int d = ks * 16 + (i >> 1) * 8 + 2 * tig;
                    qa[ks][i] = hh < group ? *reinterpret_cast<const uint32_t*>(q0 + hh * D + d) : 0u;
                }
            }
        }
        // this lane's two heads (fragment rows gid and gid + 8): running max
        // (log2 units), running sum, and O
        float m_run[2] = {-INFINITY, -INFINITY}, l_run[2] = {0.f, 0.f};
        float oc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) oc[nt][i] = 0.f;

        for (int s = it.s0; s < it.s1; ++s, ++consumed) {
            issue();
            const int st = consumed % kDecStages;
            const uint32_t sK = sRing + st * C::kStageBytes, sV = sK + C::kTileBytes;
            ok = mbar_wait(smem_u32(&bar_full[st]), (consumed / kDecStages) & 1, &abort_flag) && ok;
            if (!(ok = __all_sync(0xffffffffu, ok))) break;  // the warp leaves together (mma.sync needs all lanes)
            const int j0 = s * kDecRows + warp * kDecRowsPerWarp;  // this warp's first cache row
            if (lane < kDecRowsPerWarp) {
                // a cache row the token does not see may hold anything, NaN included:
                // zero its V so that P = 0 keeps it out of the product
                const int spos = pos_of<RING>(j0 + lane, it.len, p.R);
                const bool vis = spos >= 0 && (!RING || spos > it.len - 1 - p.window);
                if (!vis) {
                    const int row = warp * kDecRowsPerWarp + lane;
#pragma unroll
                    for (int half = 0; half < D / 64; ++half)
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch)
                            st_shared_v4(sV + half * C::kHalfBytes + sw128_offset(row, ch), 0u, 0u, 0u, 0u);
                }
            }
            __syncwarp();
            // ---- S = q.K^T over the warp's 16 rows (two 8-row tiles)
            float sc[2][4];
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) sc[nt][i] = 0.f;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                const int half = ks / 4, ch0 = (ks % 4) * 2;
                const int row = warp * kDecRowsPerWarp + (mi >> 1) * 8 + rr;
                uint32_t b0, b1, b2, b3;
                ldsm_x4(sK + half * C::kHalfBytes + sw128_offset(row, ch0 + (mi & 1)), b0, b1, b2, b3);
                mma_bf16_16816(sc[0], qa[ks], b0, b1);
                mma_bf16_16816(sc[1], qa[ks], b2, b3);
            }
            // ---- online softmax per head: c0, c1 -> head gid, c2, c3 -> head
            //      gid + 8; the 16 rows of a head sit in one lane quad
            float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
            for (int nt = 0; nt < 2; ++nt) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int spos = pos_of<RING>(j0 + nt * 8 + 2 * tig + (i & 1), it.len, p.R);
                    const bool vis = spos >= 0 && (!RING || spos > it.len - 1 - p.window);
                    sc[nt][i] = vis ? sc[nt][i] * p.scale_log2 : -INFINITY;
                    mx[i >> 1] = fmaxf(mx[i >> 1], sc[nt][i]);
                }
            }
            float alpha[2], m_use[2];
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 1));
                mx[r] = fmaxf(mx[r], __shfl_xor_sync(0xffffffffu, mx[r], 2));
                const float m_new = fmaxf(m_run[r], mx[r]);
                m_use[r] = m_new == -INFINITY ? 0.f : m_new;
                alpha[r] = ex2_approx(m_run[r] - m_use[r]);  // 0 while nothing was seen
                m_run[r] = m_new;
            }
            float ls[2] = {0.f, 0.f};
#pragma unroll
            for (int nt = 0; nt < 2; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    sc[nt][i] = ex2_approx(sc[nt][i] - m_use[i >> 1]);
                    ls[i >> 1] += sc[nt][i];
                }
#pragma unroll
            for (int r = 0; r < 2; ++r) {
                ls[r] += __shfl_xor_sync(0xffffffffu, ls[r], 1);
                ls[r] += __shfl_xor_sync(0xffffffffu, ls[r], 2);
                l_run[r] = l_run[r] * alpha[r] + ls[r];
            }
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
                oc[nt][0] *= alpha[0];
                oc[nt][1] *= alpha[0];
                oc[nt][2] *= alpha[1];
                oc[nt][3] *= alpha[1];
            }
            // P as the A fragment of rows = heads, k = the warp's 16 cache rows
            uint32_t pa[4];
            pa[0] = pack_bf16x2(sc[0][0], sc[0][1]);
            pa[1] = pack_bf16x2(sc[0][2], sc[0][3]);
            pa[2] = pack_bf16x2(sc[1][0], sc[1][1]);
            pa[3] = pack_bf16x2(sc[1][2], sc[1][3]);
            // ---- O += P.V over the warp's 16 cache rows, all D columns
#pragma unroll
            for (int np = 0; np < NT / 2; ++np) {  // pairs of 8-column tiles of V
                // matrices: (rows k0..+7, cols n), (rows k0+8..+15, cols n), then n + 8
                const int row = warp * kDecRowsPerWarp + (mi & 1) * 8 + rr;
                const int col = np * 16 + (mi >> 1) * 8;  // first head-dim column of the 16-byte chunk
                uint32_t b0, b1, b2, b3;
                ldsm_x4_trans(sV + (col / 64) * C::kHalfBytes + sw128_offset(row, (col % 64) / 8), b0, b1, b2, b3);
                mma_bf16_16816(oc[2 * np], pa, b0, b1);
                mma_bf16_16816(oc[2 * np + 1], pa, b2, b3);
            }
            // the warp is done with the stage (its V-row writes ordered before
            // the stage's next TMA write)
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bar_empty[st]));
        }
        // every thread of the CTA reaches this barrier, and all stop together if
        // any wait gave up
        if (!__syncthreads_and(ok)) break;
        // ---- the four warps' partials: [warp][head][D + 2] in shared memory
        {
            float* mw = sM + warp * group * (D + 2);
#pragma unroll
            for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int hh = gid + (i >> 1) * 8;
                    const int d = nt * 8 + 2 * tig + (i & 1);
                    if (hh < group) mw[hh * (D + 2) + d] = oc[nt][i];
                }
            }
            if (tig == 0) {
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    const int hh = gid + 8 * r;
                    if (hh < group) {
                        mw[hh * (D + 2) + D] = m_run[r];
                        mw[hh * (D + 2) + D + 1] = l_run[r];
                    }
                }
            }
        }
        __syncthreads();
        if (tid < group) {  // per head: M = max_w m_w, L = sum_w 2^(m_w - M) l_w
            float M = -INFINITY;
#pragma unroll
            for (int wv = 0; wv < 4; ++wv) M = fmaxf(M, sM[(wv * group + tid) * (D + 2) + D]);
            float L = 0.f;
#pragma unroll
            for (int wv = 0; wv < 4; ++wv) {
                const float mv = sM[(wv * group + tid) * (D + 2) + D];
                const float wgt = (M == -INFINITY || mv == -INFINITY) ? 0.f : ex2_approx(mv - M);
                sh_wm[wv][tid] = wgt;
                L += wgt * sM[(wv * group + tid) * (D + 2) + D + 1];
            }
            sh_M[tid] = M;
            sh_L[tid] = L;
        }
        __syncthreads();
        if (it.nused == 1) {  // the whole cache in this item: normalise and write the output
            for (int i = tid; i < group * D; i += kDecThreads) {
                const int hh = i / D, d = i % D;
                float acc = 0.f;
#pragma unroll
                for (int wv = 0; wv < 4; ++wv) acc += sh_wm[wv][hh] * sM[(wv * group + hh) * (D + 2) + d];
                const float L = sh_L[hh];
                const __nv_bfloat16 bv = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
                p.out[(static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * D + d] = *reinterpret_cast<const logo_bf16*>(&bv);
            }
            __syncthreads();  // the merge buffer is reused by the next item
            continue;
        }
        // ---- a chunk of a longer cache: partial result, then the last chunk merges
        for (int i = tid; i < group * D; i += kDecThreads) {
            const int hh = i / D, d = i % D;
            float acc = 0.f;
#pragma unroll
            for (int wv = 0; wv < 4; ++wv) acc += sh_wm[wv][hh] * sM[(wv * group + hh) * (D + 2) + d];
            float* dst = p.part + ((static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk + it.c) * (D + 2);
            dst[d] = acc;
            if (d == 0) {
                dst[D] = sh_M[hh];
                dst[D + 1] = sh_L[hh];
            }
        }
        __syncthreads();  // every partial of this chunk is written
        if (tid == 0) {
            __threadfence();
            const int prev = atomicAdd(p.done + static_cast<int64_t>(it.r) * p.Hkv + it.kvh, 1);
            sh_last = prev == it.nused - 1;
            if (sh_last) __threadfence();
        }
        __syncthreads();
        if (sh_last) {
            // M = max_c m_c, L = sum_c 2^(m_c - M) l_c, o = sum_c 2^(m_c - M) o_c / L,
            // per head: the weights first (into sW), then thread (head, d) adds the chunks
            for (int i = tid; i < group * it.nused; i += kDecThreads) {
                const int hh = i / it.nused;
                const float* base = p.part + (static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk * (D + 2);
                float M = -INFINITY;
                for (int c = 0; c < it.nused; ++c) M = fmaxf(M, __ldcg(base + c * (D + 2) + D));
                const int c = i % it.nused;
                const float m = __ldcg(base + c * (D + 2) + D);
                sW[hh * it.nused + c] = m == -INFINITY ? 0.f : ex2_approx(m - M);
            }
            __syncthreads();
            for (int i = tid; i < group * D; i += kDecThreads) {
                const int hh = i / D, d = i % D;
                const float* base = p.part + (static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk * (D + 2);
                const float* wts = sW + hh * it.nused;
                float o = 0.f, L = 0.f;
                for (int c = 0; c < it.nused; ++c) {
                    const float wc = wts[c];
                    o += wc * __ldcg(base + c * (D + 2) + d);
                    L += wc * __ldcg(base + c * (D + 2) + D + 1);
                }
                const __nv_bfloat16 bv = __float2bfloat16_rn(L > 0.f ? o / L : 0.f);
                p.out[(static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * D + d] = *reinterpret_cast<const logo_bf16*>(&bv);
            }
        }
        __syncthreads();  // sW and the merge buffer are reused by the next item
    }
    if (!ok && tid == 0) {  // let copies already issued land before the CTA exits
        for (int k = consumed; k < issued; ++k) mbar_wait_drain(smem_u32(&bar_full[k % kDecStages]), (k / kDecStages) & 1);
    }
}

// Chunks per (row, KV head): at least enough that a chunk holds at most
// kDecSubMax sub-tiles, more while B x Hkv items would leave SMs idle, at most
// one per sub-tile and kDecMaxChunks.  (rows: B, the most the global call can
// have selected.)
struct DecSplit {
    int nchunk, sub_per_chunk;
};

DecSplit dec_split(const logo_dims& d)
{
    const int n_sub = (d.T + kDecRows - 1) / kDecRows;
    const long long pairs = static_cast<long long>(d.B) * d.Hkv;
    const long long want = (device_sm_count() + pairs - 1) / pairs;
    long long nc = std::max<long long>(want, (n_sub + kDecSubMax - 1) / kDecSubMax);
    nc = std::min<long long>(nc, std::min(n_sub, kDecMaxChunks));
    nc = std::max<long long>(nc, 1);
    const int spc = static_cast<int>((n_sub + nc - 1) / nc);
    return DecSplit{(n_sub + spc - 1) / spc, spc};
}

// part: [B, Hq, nchunk, D + 2] fp32, then done: [B, Hkv] int32
size_t decode_ws_bytes(const logo_dims& d, size_t* done_off = nullptr)
{
    const DecSplit sp = dec_split(d);
    const size_t part = round_up(static_cast<size_t>(d.B) * d.Hq * sp.nchunk * (d.D + 2) * sizeof(float), 256);
    if (done_off) *done_off = part;
    return round_up(part + static_cast<size_t>(d.B) * d.Hkv * sizeof(int32_t), 256);
}

int check_decode(const logo_dims& d)
{
    int rc = check_dims(d);
    if (rc != LOGO_OK) return rc;
    if (d.Hq / d.Hkv > kDecMaxGroup) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

template <int D, bool RING>
int launch_decode(DecParams& prm, cudaStream_t st)
{
    static bool attr_done = false;  // benign race: setting the attribute twice is harmless
    if (!attr_done) {
        if (set_smem_limit(decode_attn_kernel<D, RING>, DecCfg<D>::smem_bytes(kDecMaxGroup)) != cudaSuccess)
            return LOGO_ERR_CUDA;
        attr_done = true;
    }
    // as many resident CTAs as fit (each keeps up to three sub-tiles' K/V loads in
    // flight); the merge buffer, and so the fit, depends on the group size
    const int group = prm.Hq / prm.Hkv;
    const int smem = DecCfg<D>::smem_bytes(group);
    static int per_sm_of[kDecMaxGroup + 1] = {};
    int per_sm = per_sm_of[group];
    if (per_sm == 0) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_attn_kernel<D, RING>, kDecThreads, smem) !=
                cudaSuccess ||
            per_sm < 1)
            per_sm = 1;
        per_sm_of[group] = per_sm;
    }
    const long long items = static_cast<long long>(prm.B) * prm.Hkv * prm.nchunk;
    const int grid = static_cast<int>(std::max(1ll, std::min(items, static_cast<long long>(per_sm) * device_sm_count())));
    if (prm.nchunk > 1 &&  // the chunk counters start at zero
        cudaMemsetAsync(prm.done, 0, static_cast<size_t>(prm.B) * prm.Hkv * sizeof(int32_t), st) != cudaSuccess)
        return LOGO_ERR_CUDA;
    decode_attn_kernel<D, RING><<<grid, kDecThreads, smem, st>>>(prm);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

int run_decode(bool ring, const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, const int32_t* seq_len,
               const int32_t* cu_q, const int32_t* n_sel, logo_bf16* out, const logo_dims& dims, int window,
               float scale, void* workspace, size_t workspace_bytes, void* stream)
{
    int rc = check_decode(dims);
    if (rc != LOGO_OK) return rc;
    if (!q || !k || !v || !seq_len || !out) return LOGO_ERR_INVALID_ARG;
    if (!ring && (!cu_q || !n_sel)) return LOGO_ERR_INVALID_ARG;
    if (ring && window < 1) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v) || !aligned16(out)) return LOGO_ERR_UNSUPPORTED;
    if (!(scale >= 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (scale == 0.0f) scale = 1.0f / sqrtf(static_cast<float>(dims.D));
    size_t done_off = 0;
    const size_t need = decode_ws_bytes(dims, &done_off);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return LOGO_ERR_WORKSPACE;
    const DecSplit sp = dec_split(dims);
    DecParams prm{};
    if (!encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kDecRows) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kDecRows))
        return LOGO_ERR_CUDA;
    prm.q = q;
    prm.seq_len = seq_len;
    prm.cu_q = cu_q;
    prm.n_sel = n_sel;
    prm.part = static_cast<float*>(workspace);
    prm.done = reinterpret_cast<int32_t*>(static_cast<char*>(workspace) + done_off);
    prm.out = out;
    prm.B = dims.B;
    prm.R = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = window;
    prm.nchunk = sp.nchunk;
    prm.sub_per_chunk = sp.sub_per_chunk;
    prm.scale_log2 = scale * kLog2e;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (dims.D == 128) return ring ? launch_decode<128, true>(prm, st) : launch_decode<128, false>(prm, st);
    return ring ? launch_decode<64, true>(prm, st) : launch_decode<64, false>(prm, st);
}

}  // namespace

int decode_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" size_t logo_decode_workspace_size(logo_dims dims)
{
    if (check_decode(dims) != LOGO_OK) return 0;
    return decode_ws_bytes(dims);
}

extern "C" int logo_decode_local_attn(const logo_bf16* q, const logo_bf16* k_ring, const logo_bf16* v_ring,
                                      const int32_t* seq_len, logo_bf16* o, logo_dims dims, int window, float scale,
                                      void* workspace, size_t workspace_bytes, void* stream)
{
    return run_decode(true, q, k_ring, v_ring, seq_len, nullptr, nullptr, o, dims, window, scale, workspace,
                      workspace_bytes, stream);
}

extern "C" int logo_decode_global_sparse_attn(const logo_bf16* q, const logo_bf16* k_cache, const logo_bf16* v_cache,
                                              const int32_t* seq_len, const int32_t* cu_q,
                                              const int32_t* n_sel_total, logo_bf16* o_c, logo_dims dims,
                                              float scale, void* workspace, size_t workspace_bytes, void* stream)
{
    return run_decode(false, q, k_cache, v_cache, seq_len, cu_q, n_sel_total, o_c, dims, kNoWindow, scale, workspace,
                      workspace_bytes, stream);
}
