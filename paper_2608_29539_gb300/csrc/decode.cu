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
// Both run one split-K kernel.  An item is 128 consecutive cache rows of one
// (row, KV head); a persistent CTA (two per SM) walks the items of the call,
// brings K and V in with TMA (128-byte swizzle) and serves every query head of
// the KV head's group from them: S = q.K^T and O = P.V as warp-level bf16
// products (mma.sync m16n8k16: the group's heads are the 16 rows, so a group
// of up to 16 heads fills one tile), the chunk's max m and sum l in log2
// units, unnormalised O.  A merge kernel combines the chunks of each
// (row, head) exactly.  Decoding is bound by HBM: every cache byte serves only
// the group's heads.  In the global call the items of rows past the
// device-side count of selected rows are never visited, so unselected
// sequences cost no cache traffic and no host synchronisation is needed.
#include <cuda_bf16.h>

#include <algorithm>
#include <cstdint>

#include "attn_common.cuh"
#include "host_common.h"
#include "logo_status.cuh"
#include "sm100.cuh"

namespace logo {
namespace {

constexpr int kDecRows = 128;     // cache rows per item (= threads per CTA, 4 warps x 32 rows)
constexpr int kDecMaxGroup = 16;  // query heads per KV head (the mma tile's 16 rows)

struct DecParams {
    CUtensorMap tm_k;  // cache [B, R, Hkv, D], box {64, 1, 128, 1}
    CUtensorMap tm_v;
    const logo_bf16* q;       // [B, Hq, D]
    const int32_t* seq_len;   // [B] tokens in the cache, the new one included
    const int32_t* cu_q;      // global: [B+1] packed rows of the (B, 1) selection
    const int32_t* n_sel;     // global: [1]
    float* part;              // [B, Hq, nchunk, D + 2]: unnormalised o, then m, l
    logo_bf16* out;           // [B, Hq, D] (global: packed rows)
    int B, R, Hq, Hkv, window, nchunk;
    float scale_log2;
};

template <int D>
struct DecCfg {
    static constexpr int kHalfBytes = kDecRows * 128;         // 64 head-dim columns of 128 rows
    static constexpr int kTileBytes = (D / 64) * kHalfBytes;  // K or V item
    static constexpr int kOffK = 0;                           // later: the warps' partial O
    static constexpr int kOffV = kTileBytes;
    static constexpr int kOffS = 2 * kTileBytes;  // [group][128] fp32 scores, then P
    static constexpr int kSmemBytes = kOffS + kDecMaxGroup * kDecRows * 4 + 1024;
    static_assert(4 * kDecMaxGroup * D * 4 <= kTileBytes, "partial O of four warps must fit in the K tile");
};

// Row j of the cache holds position pos_of(j) (or none: -1).  Dense cache:
// j itself while j < len.  Ring of R slots: the latest position congruent to j
// modulo R that is in the cache.
template <bool RING>
__device__ __forceinline__ int pos_of(int j, int len, int R)
{
    if (j >= len) return -1;
    return RING ? j + R * ((len - 1 - j) / R) : j;
}

template <int D, bool RING>
__global__ void __launch_bounds__(kDecRows, 2) decode_attn_kernel(const __grid_constant__ DecParams p)
{
    using C = DecCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_kv;
    __shared__ volatile int abort_flag;
    __shared__ float sh_m[kDecMaxGroup], sh_l[kDecMaxGroup];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int gid = lane >> 2, tig = lane & 3;  // mma fragment coordinates
    const int mi = lane >> 3, rr = lane & 7;    // ldmatrix: matrix index, row in the matrix
    const int group = p.Hq / p.Hkv;
    float* sS = reinterpret_cast<float*>(smem + C::kOffS);
    const uint32_t sK = smem_u32(smem + C::kOffK), sV = smem_u32(smem + C::kOffV);
    // rows of the call: every sequence (local), the selected packed rows (global)
    const int n_rows = RING ? p.B : *p.n_sel;
    const long long n_items = static_cast<long long>(n_rows) * p.Hkv * p.nchunk;
    if (tid == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_kv), 1);
        fence_mbar_init();
    }
    __syncthreads();
    int loads = 0;
    // persistent: items (row, KV head, chunk) in row-major order, a grid stride apart
    for (long long w = blockIdx.x; w < n_items; w += gridDim.x) {
        const int c = static_cast<int>(w % p.nchunk);
        const int t = static_cast<int>(w / p.nchunk);
        const int kvh = t % p.Hkv, r = t / p.Hkv;
        const int b = RING ? r : seq_of_row(p.cu_q, p.B, r);
        const int len = RING ? p.seq_len[b] : min(p.seq_len[b], p.R);  // a dense cache holds at most R tokens
        const int rows_used = min(len, p.R);
        const int j0 = c * kDecRows;
        if (len < 1 || j0 >= rows_used) continue;  // the merge skips chunks past the used rows
        const int h0 = kvh * group;
        if (tid == 0) {
            const uint32_t bar = smem_u32(&bar_kv);
            const uint64_t pol = policy_evict_first();
            mbar_arrive_expect_tx(bar, 2 * C::kTileBytes);
            for (int s = 0; s < D / 64; ++s) {
                tma_load_4d(sK + s * C::kHalfBytes, &p.tm_k, bar, 64 * s, kvh, j0, b, pol);
                tma_load_4d(sV + s * C::kHalfBytes, &p.tm_v, bar, 64 * s, kvh, j0, b, pol);
            }
        }
        // the group's queries as mma A fragments (rows = heads, zero past the
        // group), straight from global memory while the item loads
        uint32_t qa[D / 16][4];
        {
            const logo_bf16* q0 = p.q + (static_cast<int64_t>(b) * p.Hq + h0) * D;
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
        const bool ok = mbar_wait(smem_u32(&bar_kv), loads & 1, &abort_flag);
        ++loads;
        if (!ok) break;  // the barrier never completed for any thread: all leave here
        {
            // a cache row the token does not see may hold anything, NaN included:
            // zero its V so that P = 0 keeps it out of the product
            const int spos = pos_of<RING>(j0 + tid, len, p.R);
            const bool vis = spos >= 0 && (!RING || spos > len - 1 - p.window);
            if (!vis) {
#pragma unroll
                for (int half = 0; half < D / 64; ++half)
#pragma unroll
                    for (int ch = 0; ch < 8; ++ch)
                        st_shared_v4(sV + half * C::kHalfBytes + sw128_offset(tid, ch), 0u, 0u, 0u, 0u);
            }
        }

        // ---- S = q.K^T: warp w takes cache rows [32w, 32w + 32) (four 8-row tiles)
        {
            float sc[4][4];
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) sc[nt][i] = 0.f;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {
                const int half = ks / 4, ch0 = (ks % 4) * 2;
#pragma unroll
                for (int np = 0; np < 2; ++np) {  // pairs of 8-row tiles
                    const int row = warp * 32 + np * 16 + (mi >> 1) * 8 + rr;
                    uint32_t b0, b1, b2, b3;
                    ldsm_x4(sK + half * C::kHalfBytes + sw128_offset(row, ch0 + (mi & 1)), b0, b1, b2, b3);
                    mma_bf16_16816(sc[2 * np], qa[ks], b0, b1);
                    mma_bf16_16816(sc[2 * np + 1], qa[ks], b2, b3);
                }
            }
            // scale into log2 units, mask, store the group's rows:
            // c0, c1 -> head gid, c2, c3 -> head gid + 8
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int hh = gid + (i >> 1) * 8;
                    const int key = warp * 32 + nt * 8 + 2 * tig + (i & 1);
                    const int spos = pos_of<RING>(j0 + key, len, p.R);
                    const bool vis = spos >= 0 && (!RING || spos > len - 1 - p.window);
                    if (hh < group) sS[hh * kDecRows + key] = vis ? sc[nt][i] * p.scale_log2 : -INFINITY;
                }
            }
        }
        __syncthreads();

        // ---- per head: item max m, P = 2^(S - m) in place, sum l (a warp per head)
        for (int hh = warp; hh < group; hh += kDecRows / 32) {
            float* row = sS + hh * kDecRows;
            float v[kDecRows / 32];
            float m = -INFINITY;
#pragma unroll
            for (int i = 0; i < kDecRows / 32; ++i) {
                v[i] = row[lane + 32 * i];
                m = fmaxf(m, v[i]);
            }
            for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
            const float m_use = m == -INFINITY ? 0.f : m;
            float l = 0.f;
#pragma unroll
            for (int i = 0; i < kDecRows / 32; ++i) {
                const float e = ex2_approx(v[i] - m_use);
                row[lane + 32 * i] = e;
                l += e;
            }
            for (int o = 16; o > 0; o >>= 1) l += __shfl_xor_sync(0xffffffffu, l, o);
            if (lane == 0) {
                sh_m[hh] = m;
                sh_l[hh] = l;
            }
        }
        __syncthreads();

        // ---- O = P.V over this warp's 32 cache rows (two 16-row k-steps), all D
        //      columns; invisible rows carry P = 0 and a zeroed V row
        constexpr int NT = D / 8;
        float oc[NT][4];
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) oc[nt][i] = 0.f;
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int k0 = warp * 32 + kk * 16;
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
        __syncthreads();  // every warp is done with the K tile and with sS
        // ---- sum the four warps' partial O through shared memory (the K tile)
        float* sO = reinterpret_cast<float*>(smem + C::kOffK);  // [warp][head][D]
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
        for (int i = tid; i < group * D; i += kDecRows) {
            const int hh = i / D, d = i % D;
            float acc = 0.f;
#pragma unroll
            for (int wv = 0; wv < kDecRows / 32; ++wv) acc += sO[(wv * group + hh) * D + d];
            float* dst = p.part + ((static_cast<int64_t>(r) * p.Hq + h0 + hh) * p.nchunk + c) * (D + 2);
            dst[d] = acc;
            if (d == 0) {
                dst[D] = sh_m[hh];
                dst[D + 1] = sh_l[hh];
            }
        }
        fence_proxy_async_smem();  // thread writes to the tiles before the next item's TMA writes
        __syncthreads();           // shared memory is reused by the next item's load
    }
}

// Exact combination of the chunks of one (row, head):
// M = max m_c, L = sum l_c 2^(m_c - M), o = sum o_c 2^(m_c - M) / L.
// kMergeSplit x D threads per (row, head): a block max of the chunk maxima,
// then in batches of the block's size the chunk weights go to shared memory
// and thread (q, d) adds o_c[d] w_c over the chunks c = q (mod kMergeSplit);
// the partial sums are added in a fixed order (deterministic).  One thread
// per d walking every chunk twice left this step bound by load latency.
constexpr int kMergeSplit = 4;

template <int D, bool RING>
__global__ void __launch_bounds__(kMergeSplit * D) decode_merge_kernel(const __grid_constant__ DecParams p)
{
    constexpr int NT = kMergeSplit * D;
    __shared__ float sh_w[NT];
    __shared__ float sh_red[NT / 32];
    __shared__ float sh_o[kMergeSplit][D];
    const int r = blockIdx.x, h = blockIdx.y, t = threadIdx.x;
    const int d = t % D, q = t / D;
    int b = r;
    if (!RING) {
        if (r >= *p.n_sel) return;
        b = seq_of_row(p.cu_q, p.B, r);
    }
    const int len = RING ? p.seq_len[b] : min(p.seq_len[b], p.R);
    const int nc = (min(max(len, 0), p.R) + kDecRows - 1) / kDecRows;
    const float* base = p.part + (static_cast<int64_t>(r) * p.Hq + h) * p.nchunk * (D + 2);
    // M: strided over the threads, then warps, then the block
    float M = -INFINITY;
    for (int c = t; c < nc; c += NT) M = fmaxf(M, base[c * (D + 2) + D]);
    for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
    if ((t & 31) == 0) sh_red[t >> 5] = M;
    __syncthreads();
    M = -INFINITY;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) M = fmaxf(M, sh_red[w]);
    const float M_use = M == -INFINITY ? 0.f : M;
    float L = 0.f, o = 0.f;
    for (int c0 = 0; c0 < nc; c0 += NT) {
        __syncthreads();  // the previous batch's weights are consumed
        if (c0 + t < nc) {
            const float* pc = base + (c0 + t) * (D + 2);
            const float w = ex2_approx(pc[D] - M_use);
            sh_w[t] = w;
            L += pc[D + 1] * w;
        }
        __syncthreads();
        const int nb = min(NT, nc - c0);
#pragma unroll 4
        for (int k = q; k < nb; k += kMergeSplit) o += base[(c0 + k) * (D + 2) + d] * sh_w[k];
    }
    // L over the block (warps in order), o over the kMergeSplit lanes of each d
    for (int s2 = 16; s2 > 0; s2 >>= 1) L += __shfl_xor_sync(0xffffffffu, L, s2);
    __syncthreads();
    if ((t & 31) == 0) sh_red[t >> 5] = L;
    sh_o[q][d] = o;
    __syncthreads();
    if (q == 0) {
        float Lt = 0.f;
#pragma unroll
        for (int w = 0; w < NT / 32; ++w) Lt += sh_red[w];
        float ot = 0.f;
#pragma unroll
        for (int k = 0; k < kMergeSplit; ++k) ot += sh_o[k][d];
        const float val = Lt > 0.f ? ot / Lt : 0.f;
        const __nv_bfloat16 bv = __float2bfloat16_rn(val);
        p.out[(static_cast<int64_t>(r) * p.Hq + h) * D + d] = *reinterpret_cast<const logo_bf16*>(&bv);
    }
}

size_t decode_ws_bytes(const logo_dims& d)
{
    const int nchunk = (d.T + kDecRows - 1) / kDecRows;
    return round_up(static_cast<size_t>(d.B) * d.Hq * nchunk * (d.D + 2) * sizeof(float), 256);
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
    // as many resident CTAs as fit (each keeps one item's K/V load in flight)
    static int per_sm = 0;
    if (per_sm == 0 && (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_attn_kernel<D, RING>, kDecRows,
                                                                      DecCfg<D>::kSmemBytes) != cudaSuccess ||
                        per_sm < 1))
        per_sm = 2;
    const long long items = static_cast<long long>(prm.B) * prm.Hkv * prm.nchunk;
    const int grid = static_cast<int>(std::max(1ll, std::min(items, static_cast<long long>(per_sm) * device_sm_count())));
    decode_attn_kernel<D, RING><<<grid, kDecRows, DecCfg<D>::kSmemBytes, st>>>(prm);
    decode_merge_kernel<D, RING><<<dim3(prm.B, prm.Hq), kMergeSplit * D, 0, st>>>(prm);
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
    const size_t need = decode_ws_bytes(dims);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return LOGO_ERR_WORKSPACE;
    DecParams prm{};
    if (!encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kDecRows) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kDecRows))
        return LOGO_ERR_CUDA;
    prm.q = q;
    prm.seq_len = seq_len;
    prm.cu_q = cu_q;
    prm.n_sel = n_sel;
    prm.part = static_cast<float*>(workspace);
    prm.out = out;
    prm.B = dims.B;
    prm.R = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = window;
    prm.nchunk = (dims.T + kDecRows - 1) / kDecRows;
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
