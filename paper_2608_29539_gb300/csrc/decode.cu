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
// rows (up to kDecSubMax sub-tiles of 128 rows) of one (row, KV head); a CTA
// (4 warps) walks its items' sub-tiles through a 3-stage TMA ring (128-byte
// swizzle), so the next two sub-tiles load while one is computed, and serves
// every query head of the KV head's group from each: S = q.K^T and O = P.V as
// warp-level bf16 products (mma.sync m16n8k16: the group's heads are the 16
// rows, so a group of up to 16 heads fills one tile), with an online softmax
// (running max and sum per head, in log2 units) across the item's sub-tiles.
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
    static constexpr int kOffS = kDecStages * kStageBytes;    // [group][rows] fp32 scores, then P
    static constexpr int kSmemBytes = kOffS + kDecMaxGroup * kDecRows * 4 + 1024;
    // the warps' partial O at the end of an item go to the stage consumed last
    // (no copy targets it before the next item's first issue)
    static_assert(4 * kDecMaxGroup * D * 4 <= kStageBytes, "partial O of four warps must fit in a stage");
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
    __shared__ __align__(8) uint64_t bar_full[kDecStages];
    __shared__ volatile int abort_flag;
    __shared__ float sh_m[kDecMaxGroup], sh_l[kDecMaxGroup], sh_alpha[kDecMaxGroup];
    __shared__ int sh_last;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gid = lane >> 2, tig = lane & 3;  // mma fragment coordinates
    const int mi = lane >> 3, rr = lane & 7;    // ldmatrix: matrix index, row in the matrix
    const int group = p.Hq / p.Hkv;
    float* sS = reinterpret_cast<float*>(smem + C::kOffS);
    const uint32_t sRing = smem_u32(smem);
    // rows of the call: every sequence (local), the selected packed rows (global)
    const int n_rows = RING ? p.B : *p.n_sel;
    const long long n_items = static_cast<long long>(n_rows) * p.Hkv * p.nchunk;
    if (tid == 0) {
        abort_flag = 0;
        for (int s = 0; s < kDecStages; ++s) mbar_init(smem_u32(&bar_full[s]), 1);
        fence_mbar_init();
    }
    __syncthreads();

    // ---- the producer (thread 0) walks the same sequence of sub-tiles as the
    //      consumers, kDecStages - 1 ahead: (item w, sub-tile s) in order
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
    auto issue = [&]() {
        if (tid != 0) return;
        if (!producer_next(&pit)) return;
        const int st = issued % kDecStages;
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

    int consumed = 0;
    bool ok = true;
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
        if (tid < kDecMaxGroup) {
            sh_m[tid] = -INFINITY;
            sh_l[tid] = 0.f;
        }
        constexpr int NT = D / 8;
        float oc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) oc[nt][i] = 0.f;

        for (int s = it.s0; s < it.s1; ++s, ++consumed) {
            issue();  // the stage freed by the sub-tile before this one
            const int st = consumed % kDecStages;
            const uint32_t sK = sRing + st * C::kStageBytes, sV = sK + C::kTileBytes;
            if (!(ok = mbar_wait(smem_u32(&bar_full[st]), (consumed / kDecStages) & 1, &abort_flag))) break;
            const int j0 = s * kDecRows;
            if (tid < kDecRows) {
                // a cache row the token does not see may hold anything, NaN included:
                // zero its V so that P = 0 keeps it out of the product
                const int spos = pos_of<RING>(j0 + tid, it.len, p.R);
                const bool vis = spos >= 0 && (!RING || spos > it.len - 1 - p.window);
                if (!vis) {
#pragma unroll
                    for (int half = 0; half < D / 64; ++half)
#pragma unroll
                        for (int ch = 0; ch < 8; ++ch)
                            st_shared_v4(sV + half * C::kHalfBytes + sw128_offset(tid, ch), 0u, 0u, 0u, 0u);
                }
            }
            // ---- S = q.K^T: warp w takes cache rows [16w, 16w + 16) (two 8-row tiles)
            {
                constexpr int NTW = kDecRowsPerWarp / 8;
                float sc[NTW][4];
#pragma unroll
                for (int nt = 0; nt < NTW; ++nt)
#pragma unroll
                    for (int i = 0; i < 4; ++i) sc[nt][i] = 0.f;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const int half = ks / 4, ch0 = (ks % 4) * 2;
#pragma unroll
                    for (int np = 0; np < NTW / 2; ++np) {  // pairs of 8-row tiles
                        const int row = warp * kDecRowsPerWarp + np * 16 + (mi >> 1) * 8 + rr;
                        uint32_t b0, b1, b2, b3;
                        ldsm_x4(sK + half * C::kHalfBytes + sw128_offset(row, ch0 + (mi & 1)), b0, b1, b2, b3);
                        mma_bf16_16816(sc[2 * np], qa[ks], b0, b1);
                        mma_bf16_16816(sc[2 * np + 1], qa[ks], b2, b3);
                    }
                }
                // scale into log2 units, mask, store the group's rows:
                // c0, c1 -> head gid, c2, c3 -> head gid + 8
#pragma unroll
                for (int nt = 0; nt < NTW; ++nt) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int hh = gid + (i >> 1) * 8;
                        const int key = warp * kDecRowsPerWarp + nt * 8 + 2 * tig + (i & 1);
                        const int spos = pos_of<RING>(j0 + key, it.len, p.R);
                        const bool vis = spos >= 0 && (!RING || spos > it.len - 1 - p.window);
                        if (hh < group) sS[hh * kDecRows + key] = vis ? sc[nt][i] * p.scale_log2 : -INFINITY;
                    }
                }
            }
            __syncthreads();
            // ---- per head (a warp per head): the running max and sum, P = 2^(S - m) in place
            for (int hh = warp; hh < group; hh += kDecThreads / 32) {
                float* row = sS + hh * kDecRows;
                float v[kDecRows / 32];
                float m = -INFINITY;
#pragma unroll
                for (int i = 0; i < kDecRows / 32; ++i) {
                    v[i] = row[lane + 32 * i];
                    m = fmaxf(m, v[i]);
                }
                for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                const float m_old = sh_m[hh];
                const float m_new = fmaxf(m_old, m);
                const float m_use = m_new == -INFINITY ? 0.f : m_new;
                float l = 0.f;
#pragma unroll
                for (int i = 0; i < kDecRows / 32; ++i) {
                    const float e = ex2_approx(v[i] - m_use);
                    row[lane + 32 * i] = e;
                    l += e;
                }
                for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
                if (lane == 0) {
                    const float alpha = m_old == -INFINITY ? 0.f : ex2_approx(m_old - m_use);
                    sh_alpha[hh] = alpha;
                    sh_m[hh] = m_new;
                    sh_l[hh] = sh_l[hh] * alpha + l;
                }
            }
            __syncthreads();
            // ---- O = O * alpha + P.V over this warp's 16 cache rows (one k-step),
            //      all D columns; invisible rows carry P = 0 and a zeroed V row
            {
                const float a0 = gid < group ? sh_alpha[gid] : 1.f;
                const float a1 = gid + 8 < group ? sh_alpha[gid + 8] : 1.f;
#pragma unroll
                for (int nt = 0; nt < NT; ++nt) {
                    oc[nt][0] *= a0;
                    oc[nt][1] *= a0;
                    oc[nt][2] *= a1;
                    oc[nt][3] *= a1;
                }
            }
#pragma unroll
            for (int kk = 0; kk < kDecRowsPerWarp / 16; ++kk) {
                const int k0 = warp * kDecRowsPerWarp + kk * 16;
                uint32_t pa[4];  // P rows = heads, columns = cache rows k0..k0+15 (bf16)
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int hh = gid + (i & 1) * 8;
                    const int kc = k0 + (i >> 1) * 8 + 2 * tig;
                    float x0 = 0.f, x1 = 0.f;
                    if (hh < group) {
                        x0 = sS[hh * kDecRows + kc];
                        x1 = sS[hh * kDecRows + kc + 1];
                    }
                    pa[i] = pack_bf16x2(x0, x1);
                }
#pragma unroll
                for (int np = 0; np < NT / 2; ++np) {  // pairs of 8-column tiles of V
                    // matrices: (rows k0..+7, cols n), (rows k0+8..+15, cols n), then n + 8
                    const int row = k0 + (mi & 1) * 8 + rr;
                    const int col = np * 16 + (mi >> 1) * 8;  // first head-dim column of the 16-byte chunk
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4_trans(sV + (col / 64) * C::kHalfBytes + sw128_offset(row, (col % 64) / 8), b0, b1, b2, b3);
                    mma_bf16_16816(oc[2 * np], pa, b0, b1);
                    mma_bf16_16816(oc[2 * np + 1], pa, b2, b3);
                }
            }
            fence_proxy_async_smem();  // thread writes to the stage (V zeroing) before its next TMA write
            __syncthreads();           // the stage and sS are free for the next sub-tile
        }
        if (!ok) break;
        // ---- sum the four warps' partial O through shared memory: [warp][head][D]
        //      in the K tile of the stage consumed last
        float* sO = reinterpret_cast<float*>(smem + ((consumed - 1) % kDecStages) * C::kStageBytes);
#pragma unroll
        for (int nt = 0; nt < NT; ++nt) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int hh = gid + (i >> 1) * 8;
                const int d = nt * 8 + 2 * tig + (i & 1);
                if (hh < group) sO[(warp * group + hh) * D + d] = oc[nt][i];
            }
        }
        __syncthreads();
        if (it.nused == 1) {  // the whole cache in this item: normalise and write the output
            for (int i = tid; i < group * D; i += kDecThreads) {
                const int hh = i / D, d = i % D;
                float acc = 0.f;
#pragma unroll
                for (int wv = 0; wv < kDecThreads / 32; ++wv) acc += sO[(wv * group + hh) * D + d];
                const float L = sh_l[hh];
                const __nv_bfloat16 bv = __float2bfloat16_rn(L > 0.f ? acc / L : 0.f);
                p.out[(static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * D + d] = *reinterpret_cast<const logo_bf16*>(&bv);
            }
            __syncthreads();  // sO and sh_m / sh_l are reused by the next item
            continue;
        }
        // ---- a chunk of a longer cache: partial result, then the last chunk merges
        for (int i = tid; i < group * D; i += kDecThreads) {
            const int hh = i / D, d = i % D;
            float acc = 0.f;
#pragma unroll
            for (int wv = 0; wv < kDecThreads / 32; ++wv) acc += sO[(wv * group + hh) * D + d];
            float* dst = p.part + ((static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk + it.c) * (D + 2);
            dst[d] = acc;
            if (d == 0) {
                dst[D] = sh_m[hh];
                dst[D + 1] = sh_l[hh];
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
            // per head: the weights first (into sS), then thread (head, d) adds the chunks
            for (int i = tid; i < group * it.nused; i += kDecThreads) {
                const int hh = i / it.nused;
                const float* base = p.part + (static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk * (D + 2);
                float M = -INFINITY;
                for (int c = 0; c < it.nused; ++c) M = fmaxf(M, __ldcg(base + c * (D + 2) + D));
                const int c = i % it.nused;
                const float m = __ldcg(base + c * (D + 2) + D);
                sS[hh * it.nused + c] = m == -INFINITY ? 0.f : ex2_approx(m - M);
            }
            __syncthreads();
            for (int i = tid; i < group * D; i += kDecThreads) {
                const int hh = i / D, d = i % D;
                const float* base = p.part + (static_cast<int64_t>(it.r) * p.Hq + h0 + hh) * p.nchunk * (D + 2);
                const float* wts = sS + hh * it.nused;
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
        __syncthreads();  // sO, sS and sh_m / sh_l are reused by the next item
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
        if (set_smem_limit(decode_attn_kernel<D, RING>, DecCfg<D>::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
        attr_done = true;
    }
    // as many resident CTAs as fit (each keeps two sub-tiles' K/V loads in flight)
    static int per_sm = 0;
    if (per_sm == 0 && (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_attn_kernel<D, RING>, kDecThreads,
                                                                      DecCfg<D>::kSmemBytes) != cudaSuccess ||
                        per_sm < 1))
        per_sm = 2;
    const long long items = static_cast<long long>(prm.B) * prm.Hkv * prm.nchunk;
    const int grid = static_cast<int>(std::max(1ll, std::min(items, static_cast<long long>(per_sm) * device_sm_count())));
    if (prm.nchunk > 1 &&  // the chunk counters start at zero
        cudaMemsetAsync(prm.done, 0, static_cast<size_t>(prm.B) * prm.Hkv * sizeof(int32_t), st) != cudaSuccess)
        return LOGO_ERR_CUDA;
    decode_attn_kernel<D, RING><<<grid, kDecThreads, DecCfg<D>::kSmemBytes, st>>>(prm);
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
