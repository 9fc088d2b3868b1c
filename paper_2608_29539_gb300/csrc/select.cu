// select.cu -- logo_select: the routing decision of Eq. 7 (threshold mode) or
// the per-sequence top-k reading of the target ratio (ratio mode), and the
// stream compaction of the selected set I into the packed layout of App. B.
//
// Kernels (all on `stream`, no host synchronisation):
//   radix_select_kernel  ratio mode only: per sequence, the k-th largest gate
//                        key by 4 passes of 8-bit radix histograms; yields the
//                        threshold key and how many tokens equal to it to take.
//   count_kernel         per 1024-token chunk: tokens strictly selected and
//                        (ratio mode) tokens tied with the threshold key.
//   scan_kernel          one block: per-chunk output offsets, tie ranks,
//                        cu_q[] and the total N.
//   write_kernel         per chunk: block-wide prefix sums (warp ballots) turn
//                        the decisions into z, pos and row_of, in ascending t.
// Ratio mode with 4K < T <= 128K takes one launch instead:
//   select_ratio_cluster_kernel  one 8-CTA cluster per sequence; the CTAs share
//                        their radix histograms and counts through distributed
//                        shared memory.  Up to 4K, select_ratio_small_kernel
//                        (one block per sequence) does the same in one CTA.
#include <cooperative_groups.h>

#include <cstdint>
#include <mutex>

#include "host_common.h"
#include "logo_status.cuh"

namespace logo {
namespace {

constexpr int kChunk = 1024;     // tokens per chunk
constexpr int kThreads = 256;    // threads per chunk block, 4 tokens each
constexpr int kPerThread = kChunk / kThreads;

// Order-preserving map of a float32 gate to uint32 (larger gate -> larger
// key); -0.0 is folded onto +0.0 so the two compare equal, as floats do.
__device__ __forceinline__ uint32_t gate_key(float p)
{
    uint32_t b = __float_as_uint(p);
    if (b == 0x80000000u) b = 0u;
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

struct SeqThresh {
    uint32_t key;   // tokens with key > this are selected
    int need_eq;    // ... plus the first `need_eq` tokens with key == this
};

// Exclusive prefix sum over a 256-thread block; returns the exclusive value
// and writes the block total to *total.
__device__ __forceinline__ int block_excl_scan(int v, int* total, int* sh_warp)
{
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh_warp[warp] = x;
    __syncthreads();
    if (warp == 0) {
        int w = (lane < kThreads / 32) ? sh_warp[lane] : 0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        if (lane < kThreads / 32) sh_warp[lane] = w;  // inclusive warp totals
    }
    __syncthreads();
    int base = (warp > 0) ? sh_warp[warp - 1] : 0;
    *total = sh_warp[kThreads / 32 - 1];
    __syncthreads();
    return base + x - v;
}

// Radix histograms for 1024-thread blocks: each warp counts into its own
// copy (contention stays inside a warp however the keys cluster), then the
// copies are summed per bin.
struct WarpHist {
    int h[32][256];
};

__device__ __forceinline__ void hist_clear(WarpHist& wh)
{
    int* f = &wh.h[0][0];
    for (int i = threadIdx.x; i < 32 * 256; i += blockDim.x) f[i] = 0;
}

__device__ __forceinline__ void hist_sum(const WarpHist& wh, int* hist)
{
    for (int i = threadIdx.x; i < 256; i += blockDim.x) {
        int s = 0;
#pragma unroll 8
        for (int w = 0; w < 32; ++w) s += wh.h[w][i];
        hist[i] = s;
    }
}

// Count one key per lane into the warp's histogram (every lane of the warp
// calls this together).  The top byte of a gate's key is its sign and
// exponent, so in the first pass nearly every key of (0, 1) gates falls in one
// or two bins: there, lanes with the same bin are grouped and one atomic adds
// the group's size.  Later passes spread over many bins, and a plain atomic
// per lane is cheaper than the grouping.
__device__ __forceinline__ void count_key(WarpHist& wh, int warp, bool in, uint32_t key, int shift)
{
    const uint32_t bin = (key >> shift) & 0xFFu;
    if (shift == 24) {
        const unsigned same = __match_any_sync(0xffffffffu, in ? bin : 0x100u);
        if (in && (threadIdx.x & 31) == __ffs(same) - 1) atomicAdd(&wh.h[warp][bin], __popc(same));
    } else if (in) {
        atomicAdd(&wh.h[warp][bin], 1);
    }
}

// Warp 0: the bin holding the `remaining`-th largest key counted from the top,
// and how many keys of that bin still have to be taken (bins scanned from 255
// down, lane l holding bins 255-8l .. 248-8l).
__device__ __forceinline__ void hist_pick(const int* hist, int remaining, uint32_t prefix, int shift,
                                          uint32_t* sh_prefix, int* sh_remaining)
{
    const int lane = threadIdx.x & 31;
    int c[8], sum = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        c[i] = hist[255 - 8 * lane - i];
        sum += c[i];
    }
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    const unsigned reach = __ballot_sync(0xffffffffu, incl >= remaining);
    const int owner = reach ? __ffs(reach) - 1 : 31;
    if (lane == owner) {
        int above = incl - sum;
        int d = 255 - 8 * lane;
        for (int i = 0; i < 8; ++i, --d) {
            if (above + c[i] >= remaining || d == 0) break;
            above += c[i];
        }
        *sh_prefix = prefix | (static_cast<uint32_t>(d) << shift);
        *sh_remaining = remaining - above;
    }
}

// Ratio mode: find, per sequence, the key of the k-th largest gate.
__global__ void __launch_bounds__(1024) radix_select_kernel(const float* __restrict__ p, int T, int k,
                                                            SeqThresh* __restrict__ out)
{
    __shared__ WarpHist wh;
    __shared__ int hist[256];
    __shared__ uint32_t sh_prefix;
    __shared__ int sh_remaining;
    const int b = blockIdx.x, warp = threadIdx.x >> 5;
    const float* pb = p + static_cast<int64_t>(b) * T;
    if (k <= 0) {
        if (threadIdx.x == 0) out[b] = SeqThresh{0xFFFFFFFFu, 0};
        return;
    }
    if (k >= T) {
        if (threadIdx.x == 0) out[b] = SeqThresh{0u, T};
        return;
    }
    uint32_t prefix = 0, mask = 0;
    int remaining = k;
    for (int shift = 24; shift >= 0; shift -= 8) {
        hist_clear(wh);
        __syncthreads();
        // eight loads per thread in flight before the counting
        for (int base = 0; base < T; base += 8 * blockDim.x) {
            uint32_t keys[8];
            bool valid[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) {
                const int t = base + u * blockDim.x + threadIdx.x;
                valid[u] = t < T;
                keys[u] = valid[u] ? gate_key(pb[t]) : 0u;
            }
#pragma unroll
            for (int u = 0; u < 8; ++u) count_key(wh, warp, valid[u] && (keys[u] & mask) == prefix, keys[u], shift);
        }
        __syncthreads();
        hist_sum(wh, hist);
        __syncthreads();
        if (warp == 0) hist_pick(hist, remaining, prefix, shift, &sh_prefix, &sh_remaining);
        __syncthreads();
        prefix = sh_prefix;
        remaining = sh_remaining;
        mask |= 0xFFu << shift;
        __syncthreads();
    }
    if (threadIdx.x == 0) out[b] = SeqThresh{prefix, remaining};
}

// Ratio mode, T <= 1024 * KPT: the whole selection of one sequence in one
// block of 1024 threads.  Every sequence selects exactly k_eff tokens, so
// sequence b's packed rows start at b * k_eff and no scan across sequences is
// needed.  A thread owns KPT consecutive tokens (keys kept in registers for
// the four radix passes), so block-wide scans in thread order are scans in t.
// The gates come in, and z / row_of go out, through shared memory with
// coalesced accesses (a thread's own tokens are KPT words apart from its
// neighbours': read or written straight from global memory they cost one
// sector per lane per access on the block's single SM).
template <int KPT>
__global__ void __launch_bounds__(1024) select_ratio_small_kernel(const float* __restrict__ p, int B, int T, int k,
                                                                  uint8_t* __restrict__ z, int32_t* __restrict__ pos,
                                                                  int32_t* __restrict__ cu_q,
                                                                  int32_t* __restrict__ row_of,
                                                                  int32_t* __restrict__ n_total)
{
    // [T + T/16] keys, then row_of, one pad word after every 16 (a thread's 16
    // words start on a different bank for each lane); [T] positions of the
    // selected tokens; [T] bytes of z
    extern __shared__ uint32_t stage[];
    int* pos_st = reinterpret_cast<int*>(stage + T + T / 16 + 1);
    uint8_t* zst = reinterpret_cast<uint8_t*>(pos_st + T);
    auto pad = [](int i) { return i + (i >> 4); };
    __shared__ WarpHist wh;
    __shared__ int hist[256];
    __shared__ uint32_t sh_prefix;
    __shared__ int sh_remaining;
    __shared__ int sh_warp[32];
    const int b = blockIdx.x, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t off = static_cast<int64_t>(b) * T;
    const int t0 = threadIdx.x * KPT;
    {
        float g[KPT];  // all of a thread's loads in flight at once
#pragma unroll
        for (int u = 0; u < KPT; ++u) {
            const int i = threadIdx.x + u * 1024;
            g[u] = i < T ? p[off + i] : 0.f;
        }
#pragma unroll
        for (int u = 0; u < KPT; ++u) {
            const int i = threadIdx.x + u * 1024;
            if (i < T) stage[pad(i)] = gate_key(g[u]);
        }
    }
    __syncthreads();
    uint32_t key[KPT];
    bool valid[KPT];
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        valid[u] = t0 + u < T;
        key[u] = valid[u] ? stage[pad(t0 + u)] : 0u;
    }
    // the k-th largest key, as radix_select_kernel finds it
    const int k_eff = k <= 0 ? 0 : (k >= T ? T : k);
    uint32_t prefix = 0;
    int remaining = k;
    if (k <= 0) {
        prefix = 0xFFFFFFFFu;
        remaining = 0;
    } else if (k >= T) {
        prefix = 0u;
        remaining = T;
    } else {
        uint32_t mask = 0;
        for (int shift = 24; shift >= 0; shift -= 8) {
            hist_clear(wh);
            __syncthreads();
#pragma unroll
            for (int u = 0; u < KPT; ++u) count_key(wh, warp, valid[u] && (key[u] & mask) == prefix, key[u], shift);
            __syncthreads();
            hist_sum(wh, hist);
            __syncthreads();
            if (warp == 0) hist_pick(hist, remaining, prefix, shift, &sh_prefix, &sh_remaining);
            __syncthreads();
            prefix = sh_prefix;
            remaining = sh_remaining;
            mask |= 0xFFu << shift;
            __syncthreads();
        }
    }
    // decisions: above the k-th key, plus the first `remaining` tokens equal to it
    int neq = 0;
#pragma unroll
    for (int u = 0; u < KPT; ++u) neq += (valid[u] && key[u] == prefix) ? 1 : 0;
    auto block_scan = [&](int v) {  // exclusive scan over the 1024 threads in order
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) sh_warp[warp] = x;
        __syncthreads();
        if (warp == 0) {
            int w = sh_warp[lane];
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            sh_warp[lane] = w - sh_warp[lane];  // exclusive over warps
        }
        __syncthreads();
        const int r = sh_warp[warp] + x - v;
        __syncthreads();
        return r;
    };
    int eq_rank = block_scan(neq);
    bool sel[KPT];
    int nsel = 0;
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        bool take = false;
        if (valid[u] && key[u] == prefix) {
            take = eq_rank < remaining;
            ++eq_rank;
        }
        sel[u] = valid[u] && (key[u] > prefix || take);
        nsel += sel[u];
    }
    int lrow = block_scan(nsel);  // its barriers also end every read of the staged keys
    int* row_st = reinterpret_cast<int*>(stage);
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        if (valid[u]) {
            zst[t0 + u] = sel[u] ? 1 : 0;
            row_st[pad(t0 + u)] = sel[u] ? b * k_eff + lrow : -1;
            if (sel[u]) pos_st[lrow++] = t0 + u;
        }
    }
    __syncthreads();
    for (int i = threadIdx.x; i < k_eff; i += blockDim.x) pos[static_cast<int64_t>(b) * k_eff + i] = pos_st[i];
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        const int i = threadIdx.x + u * 1024;
        if (i < T) {
            z[off + i] = zst[i];
            row_of[off + i] = row_st[pad(i)];
        }
    }
    if (threadIdx.x == 0) {
        cu_q[b] = b * k_eff;
        if (b == B - 1) {
            cu_q[B] = B * k_eff;
            *n_total = B * k_eff;
        }
    }
}

// Ratio mode, 4K < T <= kClusterCTAs * 1024 * KPT: one cluster of kClusterCTAs
// CTAs per sequence (a thread-block cluster; grid = B clusters).  CTA r of the
// cluster owns tokens [r C, r C + C), C = ceil(T / kClusterCTAs), thread i of it
// the KPT consecutive tokens starting at r C + KPT i, kept in registers.  Each
// radix pass counts the CTA's own keys into its 256-bin histogram (lanes with
// the same bin grouped, one shared atomic per group), then every CTA sums all
// kClusterCTAs histograms out of distributed shared memory, in rank order, and
// picks the same bin.  Histograms alternate between two buffers, so one
// cluster barrier per pass suffices: a buffer is cleared right after the
// barrier that follows its last remote read.  Finally the CTAs exchange their
// counts of keys above and equal to the threshold: tied keys are taken in
// position order, so a CTA's first tied rank and its first packed row follow
// from the counts of the CTAs before it.  Same decisions as the one-block
// kernel, bit for bit.
constexpr int kClusterCTAs = 8;

template <int KPT>
__global__ void __cluster_dims__(kClusterCTAs, 1, 1) __launch_bounds__(1024)
    select_ratio_cluster_kernel(const float* __restrict__ p, int B, int T, int k, uint8_t* __restrict__ z,
                                int32_t* __restrict__ pos, int32_t* __restrict__ cu_q,
                                int32_t* __restrict__ row_of, int32_t* __restrict__ n_total)
{
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    __shared__ int hist[2][256];        // this CTA's histogram of the pass (two buffers, read by the cluster)
    __shared__ int ghist[256];          // the cluster's histogram of the pass
    __shared__ int counts[2];           // keys above / equal to the threshold in this CTA (read by the cluster)
    __shared__ uint32_t sh_prefix;
    __shared__ int sh_remaining;
    __shared__ int sh_warp[32];
    __shared__ int sh_total;
    const int rank = static_cast<int>(cluster.block_rank());
    const int b = blockIdx.x / kClusterCTAs, lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t off = static_cast<int64_t>(b) * T;
    const int C = (T + kClusterCTAs - 1) / kClusterCTAs;
    const int c0 = rank * C, c1 = min(T, c0 + C);
    const int t0 = c0 + threadIdx.x * KPT;
    uint32_t key[KPT];
    bool valid[KPT];
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        valid[u] = t0 + u < c1;
        key[u] = valid[u] ? gate_key(p[off + t0 + u]) : 0u;
    }
    if (threadIdx.x < 256) {
        hist[0][threadIdx.x] = 0;
        hist[1][threadIdx.x] = 0;
    }
    __syncthreads();
    const int k_eff = k <= 0 ? 0 : (k >= T ? T : k);
    uint32_t prefix = 0;
    int remaining = k;
    if (k <= 0) {
        prefix = 0xFFFFFFFFu;
        remaining = 0;
    } else if (k >= T) {
        prefix = 0u;
        remaining = T;
    } else {
        uint32_t mask = 0;
        int buf = 0;
        for (int shift = 24; shift >= 0; shift -= 8, buf ^= 1) {
#pragma unroll
            for (int u = 0; u < KPT; ++u) {
                const bool in = valid[u] && (key[u] & mask) == prefix;
                const uint32_t bin = (key[u] >> shift) & 0xFFu;
                const unsigned same = __match_any_sync(0xffffffffu, in ? bin : 0x100u);
                if (in && lane == __ffs(same) - 1) atomicAdd(&hist[buf][bin], __popc(same));
            }
            cluster.sync();  // every CTA's histogram of this pass is complete
            if (threadIdx.x < 256) {
                int sum = 0;
                for (int r = 0; r < kClusterCTAs; ++r) sum += cluster.map_shared_rank(&hist[buf][0], r)[threadIdx.x];
                ghist[threadIdx.x] = sum;
                // the other buffer was last read remotely before the barrier above
                hist[buf ^ 1][threadIdx.x] = 0;
            }
            __syncthreads();
            if (warp == 0) hist_pick(ghist, remaining, prefix, shift, &sh_prefix, &sh_remaining);
            __syncthreads();
            prefix = sh_prefix;
            remaining = sh_remaining;
            mask |= 0xFFu << shift;
        }
    }
    // exclusive scan over the CTA's 1024 threads in order; the total to every thread
    auto block_scan = [&](int v, int* total) {
        int x = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, x, o);
            if (lane >= o) x += y;
        }
        if (lane == 31) sh_warp[warp] = x;
        __syncthreads();
        if (warp == 0) {
            const int w0 = sh_warp[lane];
            int w = w0;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int y = __shfl_up_sync(0xffffffffu, w, o);
                if (lane >= o) w += y;
            }
            sh_warp[lane] = w - w0;  // exclusive over warps
            if (lane == 31) sh_total = w;
        }
        __syncthreads();
        const int r = sh_warp[warp] + x - v;
        *total = sh_total;
        __syncthreads();
        return r;
    };
    // this CTA's keys above the threshold (low 16 bits) and tied with it (high
    // 16 bits; at most 16K per CTA), scanned together
    int ngt = 0, neq = 0;
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        ngt += (valid[u] && key[u] > prefix) ? 1 : 0;
        neq += (valid[u] && key[u] == prefix) ? 1 : 0;
    }
    int tot;
    const int ex = block_scan(ngt | (neq << 16), &tot);
    int eq_rank = ex >> 16;
    if (threadIdx.x == 0) {
        counts[0] = tot & 0xFFFF;
        counts[1] = tot >> 16;
    }
    cluster.sync();  // every CTA's counts are published
    // tied keys in earlier CTAs, and the packed rows the earlier CTAs fill
    int eq_before = 0, rows_before = 0;
    for (int r = 0; r < rank; ++r) {
        const int* rc = cluster.map_shared_rank(&counts[0], r);
        const int gt_r = rc[0], eq_r = rc[1];
        rows_before += gt_r + max(0, min(eq_r, remaining - eq_before));
        eq_before += eq_r;
    }
    eq_rank += eq_before;
    bool sel[KPT];
    int nsel = 0;
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        bool take = false;
        if (valid[u] && key[u] == prefix) {
            take = eq_rank < remaining;
            ++eq_rank;
        }
        sel[u] = valid[u] && (key[u] > prefix || take);
        nsel += sel[u];
    }
    int tot_sel;
    int row = b * k_eff + rows_before + block_scan(nsel, &tot_sel);
#pragma unroll
    for (int u = 0; u < KPT; ++u) {
        if (valid[u]) {
            z[off + t0 + u] = sel[u] ? 1 : 0;
            row_of[off + t0 + u] = sel[u] ? row : -1;
            if (sel[u]) pos[row++] = t0 + u;
        }
    }
    if (rank == 0 && threadIdx.x == 0) {
        cu_q[b] = b * k_eff;
        if (b == B - 1) {
            cu_q[B] = B * k_eff;
            *n_total = B * k_eff;
        }
    }
    cluster.sync();  // no CTA leaves while another may still read its counts
}

struct ChunkCounts {
    int gt;   // tokens selected outright in the chunk
    int eq;   // tokens tied with the threshold key (ratio mode)
};

__device__ __forceinline__ void decide(float pv, bool ratio_mode, float b_th, const SeqThresh& th, bool* gt,
                                       bool* eq)
{
    if (ratio_mode) {
        uint32_t key = gate_key(pv);
        *gt = key > th.key;
        *eq = key == th.key;
    } else {
        *gt = pv > b_th;  // Eq. 7, strict
        *eq = false;
    }
}

__global__ void __launch_bounds__(kThreads) count_kernel(const float* __restrict__ p, int T, int nchunk,
                                                         int ratio_mode, float b_th_host,
                                                         const float* __restrict__ b_th_dev,
                                                         const SeqThresh* __restrict__ th,
                                                         ChunkCounts* __restrict__ counts)
{
    __shared__ int sh_warp[kThreads / 32];
    const int c = blockIdx.x, b = blockIdx.y;
    const int t0 = c * kChunk + threadIdx.x * kPerThread;
    const float* pb = p + static_cast<int64_t>(b) * T;
    SeqThresh tb = ratio_mode ? th[b] : SeqThresh{0u, 0};
    const float b_th = b_th_dev ? *b_th_dev : b_th_host;  // Eq. 7 threshold (device-resident if given)
    int ngt = 0, neq = 0;
#pragma unroll
    for (int i = 0; i < kPerThread; ++i) {
        int t = t0 + i;
        if (t < T) {
            bool gt, eq;
            decide(pb[t], ratio_mode, b_th, tb, &gt, &eq);
            ngt += gt;
            neq += eq;
        }
    }
    int tot_gt, tot_eq;
    block_excl_scan(ngt, &tot_gt, sh_warp);
    block_excl_scan(neq, &tot_eq, sh_warp);
    if (threadIdx.x == 0) counts[static_cast<int64_t>(b) * nchunk + c] = ChunkCounts{tot_gt, tot_eq};
}

struct ChunkPlan {
    int out_base;  // packed row of the chunk's first selected token
    int eq_before; // tied tokens in earlier chunks of the same sequence
};

// One block: turns chunk counts into packed offsets (batch-major, ascending
// t) and tie ranks; writes cu_q[0..B] and the total.
__global__ void __launch_bounds__(kThreads) scan_kernel(const ChunkCounts* __restrict__ counts, int B, int nchunk,
                                                        int ratio_mode, const SeqThresh* __restrict__ th,
                                                        ChunkPlan* __restrict__ plan, int32_t* __restrict__ cu_q,
                                                        int32_t* __restrict__ n_total)
{
    __shared__ int sh_warp[kThreads / 32];
    int carry = 0;
    for (int b = 0; b < B; ++b) {
        if (threadIdx.x == 0) cu_q[b] = carry;
        const int need = ratio_mode ? th[b].need_eq : 0;
        int eq_carry = 0;
        for (int c0 = 0; c0 < nchunk; c0 += kThreads) {
            const int c = c0 + threadIdx.x;
            ChunkCounts cc = (c < nchunk) ? counts[static_cast<int64_t>(b) * nchunk + c] : ChunkCounts{0, 0};
            int eq_tot;
            int eq_before = eq_carry + block_excl_scan(cc.eq, &eq_tot, sh_warp);
            int take_eq = ratio_mode ? max(0, min(cc.eq, need - eq_before)) : 0;
            int sel = cc.gt + take_eq;
            int sel_tot;
            int base = carry + block_excl_scan(sel, &sel_tot, sh_warp);
            if (c < nchunk) plan[static_cast<int64_t>(b) * nchunk + c] = ChunkPlan{base, eq_before};
            carry += sel_tot;
            eq_carry += eq_tot;
        }
    }
    if (threadIdx.x == 0) {
        cu_q[B] = carry;
        *n_total = carry;
    }
}

__global__ void __launch_bounds__(kThreads) write_kernel(const float* __restrict__ p, int T, int nchunk,
                                                         int ratio_mode, float b_th_host,
                                                         const float* __restrict__ b_th_dev,
                                                         const SeqThresh* __restrict__ th,
                                                         const ChunkPlan* __restrict__ plan,
                                                         uint8_t* __restrict__ z, int32_t* __restrict__ pos,
                                                         int32_t* __restrict__ row_of)
{
    __shared__ int sh_warp[kThreads / 32];
    const int c = blockIdx.x, b = blockIdx.y;
    const int t0 = c * kChunk + threadIdx.x * kPerThread;
    const int64_t off = static_cast<int64_t>(b) * T;
    SeqThresh tb = ratio_mode ? th[b] : SeqThresh{0u, 0};
    const float b_th = b_th_dev ? *b_th_dev : b_th_host;
    ChunkPlan pl = plan[static_cast<int64_t>(b) * nchunk + c];
    bool gt[kPerThread], eq[kPerThread];
    int neq = 0;
#pragma unroll
    for (int i = 0; i < kPerThread; ++i) {
        int t = t0 + i;
        gt[i] = eq[i] = false;
        if (t < T) decide(p[off + t], ratio_mode, b_th, tb, &gt[i], &eq[i]);
        neq += eq[i];
    }
    int tot;
    int eq_rank = pl.eq_before + block_excl_scan(neq, &tot, sh_warp);
    bool sel[kPerThread];
    int nsel = 0;
#pragma unroll
    for (int i = 0; i < kPerThread; ++i) {
        bool take = false;
        if (eq[i]) {
            take = eq_rank < tb.need_eq;
            ++eq_rank;
        }
        sel[i] = gt[i] || take;
        nsel += sel[i];
    }
    int row = pl.out_base + block_excl_scan(nsel, &tot, sh_warp);
#pragma unroll
    for (int i = 0; i < kPerThread; ++i) {
        int t = t0 + i;
        if (t < T) {
            z[off + t] = sel[i] ? 1 : 0;
            row_of[off + t] = sel[i] ? row : -1;
            if (sel[i]) pos[row++] = t;
        }
    }
}

struct SelectWs {
    SeqThresh* th;
    ChunkCounts* counts;
    ChunkPlan* plan;
};

size_t select_ws_layout(const logo_dims& d, char* base, SelectWs* ws)
{
    const size_t nchunk = (static_cast<size_t>(d.T) + kChunk - 1) / kChunk;
    size_t off = 0;
    size_t th_off = off;
    off = round_up(off + sizeof(SeqThresh) * d.B, 256);
    size_t cnt_off = off;
    off = round_up(off + sizeof(ChunkCounts) * d.B * nchunk, 256);
    size_t plan_off = off;
    off = round_up(off + sizeof(ChunkPlan) * d.B * nchunk, 256);
    if (ws) {
        ws->th = reinterpret_cast<SeqThresh*>(base + th_off);
        ws->counts = reinterpret_cast<ChunkCounts*>(base + cnt_off);
        ws->plan = reinterpret_cast<ChunkPlan*>(base + plan_off);
    }
    return off;
}

}  // namespace

int select_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" size_t logo_select_workspace_size(logo_dims dims)
{
    if (dims.B < 1 || dims.T < 1) return 0;
    return select_ws_layout(dims, nullptr, nullptr);
}

extern "C" int logo_select(const float* gate_p, logo_dims dims, int mode, float b_th, float ratio, uint8_t* z,
                           int32_t* pos, int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total, void* workspace,
                           size_t workspace_bytes, void* stream)
{
    if (dims.B < 1 || dims.T < 1) return LOGO_ERR_INVALID_ARG;
    if (static_cast<int64_t>(dims.B) * dims.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    if (!gate_p || !z || !pos || !cu_q || !row_of || !n_sel_total) return LOGO_ERR_INVALID_ARG;
    if (mode != LOGO_SELECT_THRESHOLD && mode != LOGO_SELECT_RATIO) return LOGO_ERR_INVALID_ARG;
    const bool ratio_mode = (mode == LOGO_SELECT_RATIO);
    if (ratio_mode && !(ratio >= 0.0f && ratio <= 1.0f)) return LOGO_ERR_INVALID_ARG;
    const size_t need = select_ws_layout(dims, nullptr, nullptr);
    if (!workspace || workspace_bytes < need) return LOGO_ERR_WORKSPACE;
    SelectWs ws;
    select_ws_layout(dims, static_cast<char*>(workspace), &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int nchunk = (dims.T + kChunk - 1) / kChunk;
    // k = floor(rho * T), with rho read as float32 and the product in double
    const int k = ratio_mode ? static_cast<int>(static_cast<double>(ratio) * dims.T) : 0;
    if (ratio_mode && dims.T <= 4 * 1024) {  // one launch: one block per sequence
        const int smem =
            static_cast<int>(round_up((static_cast<size_t>(dims.T) + dims.T / 16 + 1 + dims.T) * 4 + dims.T, 16));
        if (set_smem_limit(select_ratio_small_kernel<4>, smem) != cudaSuccess) return LOGO_ERR_CUDA;
        select_ratio_small_kernel<4><<<dims.B, 1024, smem, st>>>(gate_p, dims.B, dims.T, k, z, pos, cu_q, row_of,
                                                                 n_sel_total);
        return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
    }
    if (ratio_mode && dims.T <= kClusterCTAs * 1024 * 16) {  // one launch: one 8-CTA cluster per sequence
        const dim3 grid(dims.B * kClusterCTAs);
        const int per_cta = (dims.T + kClusterCTAs - 1) / kClusterCTAs;
        if (per_cta <= 2 * 1024)
            select_ratio_cluster_kernel<2><<<grid, 1024, 0, st>>>(gate_p, dims.B, dims.T, k, z, pos, cu_q, row_of,
                                                                  n_sel_total);
        else if (per_cta <= 4 * 1024)
            select_ratio_cluster_kernel<4><<<grid, 1024, 0, st>>>(gate_p, dims.B, dims.T, k, z, pos, cu_q, row_of,
                                                                  n_sel_total);
        else if (per_cta <= 8 * 1024)
            select_ratio_cluster_kernel<8><<<grid, 1024, 0, st>>>(gate_p, dims.B, dims.T, k, z, pos, cu_q, row_of,
                                                                  n_sel_total);
        else
            select_ratio_cluster_kernel<16><<<grid, 1024, 0, st>>>(gate_p, dims.B, dims.T, k, z, pos, cu_q, row_of,
                                                                   n_sel_total);
        return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
    }
    if (ratio_mode) radix_select_kernel<<<dims.B, 1024, 0, st>>>(gate_p, dims.T, k, ws.th);
    dim3 grid(nchunk, dims.B);
    count_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, ratio_mode, b_th, nullptr, ws.th, ws.counts);
    scan_kernel<<<1, kThreads, 0, st>>>(ws.counts, dims.B, nchunk, ratio_mode, ws.th, ws.plan, cu_q, n_sel_total);
    write_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, ratio_mode, b_th, nullptr, ws.th, ws.plan, z, pos,
                                            row_of);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

// Threshold mode with b_th read from device memory by the kernels, so that a
// device-side budget controller (logo_budget_update, Eq. 11) can move the
// threshold between steps without a host round trip.
extern "C" int logo_select_device_threshold(const float* gate_p, logo_dims dims, const float* b_th, uint8_t* z,
                                            int32_t* pos, int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total,
                                            void* workspace, size_t workspace_bytes, void* stream)
{
    if (dims.B < 1 || dims.T < 1) return LOGO_ERR_INVALID_ARG;
    if (static_cast<int64_t>(dims.B) * dims.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    if (!gate_p || !b_th || !z || !pos || !cu_q || !row_of || !n_sel_total) return LOGO_ERR_INVALID_ARG;
    const size_t need = select_ws_layout(dims, nullptr, nullptr);
    if (!workspace || workspace_bytes < need) return LOGO_ERR_WORKSPACE;
    SelectWs ws;
    select_ws_layout(dims, static_cast<char*>(workspace), &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int nchunk = (dims.T + kChunk - 1) / kChunk;
    dim3 grid(nchunk, dims.B);
    count_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, 0, 0.0f, b_th, ws.th, ws.counts);
    scan_kernel<<<1, kThreads, 0, st>>>(ws.counts, dims.B, nchunk, 0, ws.th, ws.plan, cu_q, n_sel_total);
    write_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, 0, 0.0f, b_th, ws.th, ws.plan, z, pos, row_of);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

// ---------------------------------------------------------------------------
// logo_select_noalloc: the same kernels with their scratch in a static device
// array instead of a caller workspace (for callers that cannot allocate).
namespace logo {
namespace {

static __device__ __align__(256) unsigned char g_select_noalloc_scratch[LOGO_SELECT_NOALLOC_SCRATCH_BYTES];

// Id of the calling thread's current CUDA context (0 when there is none yet
// or the driver cannot tell), through the driver entry points, so the
// library keeps no link-time dependency on libcuda.
unsigned long long current_context_id()
{
    typedef CUresult (*GetCurrentFn)(CUcontext*);
    typedef CUresult (*GetIdFn)(CUcontext, unsigned long long*);
    static GetCurrentFn get_current = nullptr;
    static GetIdFn get_id = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_current = reinterpret_cast<GetCurrentFn>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<GetIdFn>(p);
    });
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS)
        return 0;
    return id;
}

// Device address of the array in the current context (the name is only a
// host-side stand-in and must never be passed to a kernel).  Looked up on the
// first call in each context and cached under the context's id, so a context
// that was destroyed and created again (cudaDeviceReset) gets a fresh lookup
// instead of a stale address.  Without a context id the lookup is repeated on
// every call.
int noalloc_scratch_ptr(char** out)
{
    static std::mutex mu;
    static unsigned long long cached_ctx[64] = {0};
    static void* cached_ptr[64] = {nullptr};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return LOGO_ERR_CUDA;
    std::lock_guard<std::mutex> lock(mu);
    const unsigned long long ctx = current_context_id();
    if (ctx != 0 && ctx == cached_ctx[dev] && cached_ptr[dev]) {
        *out = static_cast<char*>(cached_ptr[dev]);
        return LOGO_OK;
    }
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_select_noalloc_scratch) != cudaSuccess || !p) return LOGO_ERR_CUDA;
    cached_ctx[dev] = current_context_id();  // the lookup creates the context if there was none
    cached_ptr[dev] = p;
    *out = static_cast<char*>(p);
    return LOGO_OK;
}

}  // namespace
}  // namespace logo

extern "C" int logo_select_noalloc(const float* gate_p, logo_dims dims, int mode, float b_th, float ratio,
                                   uint8_t* z, int32_t* pos, int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total,
                                   void* stream)
{
    if (dims.B < 1 || dims.T < 1) return LOGO_ERR_INVALID_ARG;
    if (!gate_p || !z || !pos || !cu_q || !row_of || !n_sel_total) return LOGO_ERR_INVALID_ARG;
    if (mode != LOGO_SELECT_THRESHOLD && mode != LOGO_SELECT_RATIO) return LOGO_ERR_INVALID_ARG;
    const bool ratio_mode = (mode == LOGO_SELECT_RATIO);
    if (ratio_mode && !(ratio >= 0.0f && ratio <= 1.0f)) return LOGO_ERR_INVALID_ARG;
    const int64_t nchunk64 = (static_cast<int64_t>(dims.T) + kChunk - 1) / kChunk;
    if (dims.B > LOGO_SELECT_NOALLOC_MAX_SEQS || dims.B * nchunk64 > LOGO_SELECT_NOALLOC_MAX_CHUNKS)
        return LOGO_ERR_SCRATCH_LIMIT;
    if (select_ws_layout(dims, nullptr, nullptr) > sizeof(g_select_noalloc_scratch)) return LOGO_ERR_SCRATCH_LIMIT;
    char* scratch = nullptr;
    int rc = noalloc_scratch_ptr(&scratch);
    if (rc != LOGO_OK) return rc;
    SelectWs ws;
    select_ws_layout(dims, scratch, &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int nchunk = static_cast<int>(nchunk64);
    const int k = ratio_mode ? static_cast<int>(static_cast<double>(ratio) * dims.T) : 0;
    if (ratio_mode) radix_select_kernel<<<dims.B, 1024, 0, st>>>(gate_p, dims.T, k, ws.th);
    dim3 grid(nchunk, dims.B);
    count_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, ratio_mode, b_th, nullptr, ws.th, ws.counts);
    scan_kernel<<<1, kThreads, 0, st>>>(ws.counts, dims.B, nchunk, ratio_mode, ws.th, ws.plan, cu_q, n_sel_total);
    write_kernel<<<grid, kThreads, 0, st>>>(gate_p, dims.T, nchunk, ratio_mode, b_th, nullptr, ws.th, ws.plan, z, pos,
                                            row_of);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
