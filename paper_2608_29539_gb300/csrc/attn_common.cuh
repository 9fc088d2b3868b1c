// attn_common.cuh -- pieces shared by the attention forward and backward
// kernels: tile geometry, work-item decoding for the local (Eq. 6) and the
// query-sparse global (Eq. 8) branches, and the row/key visibility rule.
#pragma once
#include <cuda.h>

#include <cstdint>

#include "../../include/logo.h"

namespace logo {

constexpr int kBM = 128;              // query rows per tile (TMEM lanes)
constexpr int kBN = 128;              // keys per KV block
constexpr int kNoWindow = 1 << 30;    // "window" of the global branch (C^inf_t)
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

// One schedule entry of the global branch: a tile of up to 128 packed rows of
// one sequence, the range of real positions it covers (App. B: the KV blocks
// before min_pos need no causal predicate, those after max_pos none at all),
// and the KV blocks this entry visits: all of [0, max_pos / 128], or, when the
// tiles are too few to fill the GPU, one share of that range whose partial
// softmax result goes to a slot that a merge kernel combines with the others.
struct GlobalTile {
    int row0;     // first packed row
    int nrows;    // rows in the tile (1..128)
    int b;        // sequence
    int min_pos;  // position of the first row
    int max_pos;  // position of the last row
    int blk_lo;   // KV blocks visited (inclusive)
    int blk_hi;
    int slot;     // -1: the whole range, output written directly; else the partial-result slot
    int cost;     // KV blocks visited (the ordering key)
    int pad0, pad1, pad2;
};

// A tile whose KV range is split: the merge kernel combines slots
// slot0 .. slot0 + nsplit - 1 into its output rows.
struct SplitTile {
    int row0, nrows, slot0, nsplit;
};

// Everything the roles of a forward CTA need to know about one work item.
struct FwdItem {
    int b, h, kvh;
    int row0;       // local: first query position; global: first packed row
    int nrows;      // valid rows
    int pos_min, pos_max;
    int blk_lo, blk_hi;  // inclusive KV block range
    int slot;            // global split entry: partial-result slot; otherwise -1
};

// Does KV block n need the per-element visibility test for any row of the
// item?  Rows see keys s with pos - W < s <= pos.
__device__ __forceinline__ bool block_needs_mask(int n, int pos_min, int pos_max, int window)
{
    const int k0 = n * kBN, k1 = n * kBN + kBN - 1;
    return !(k1 <= pos_min && k0 > pos_max - window);
}

__device__ __forceinline__ bool key_visible(int key, int pos, int window)
{
    return key <= pos && key > pos - window;
}

// Sequence of packed row `row`: the b with cu_q[b] <= row < cu_q[b+1].
__device__ __forceinline__ int seq_of_row(const int32_t* cu_q, int B, int row)
{
    int lo = 0, hi = B - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (cu_q[mid] <= row) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

// Gather the selected rows of the dense Q into the packed layout (App. B) and
// zero the 128 rows after the last one, so that a partial final tile reads
// finite values.
static __global__ void __launch_bounds__(256)
    gather_rows_kernel(const logo_bf16* __restrict__ q, const int32_t* __restrict__ pos,
                       const int32_t* __restrict__ cu_q, const int32_t* __restrict__ n_sel, int B, int T,
                       int row_elems, logo_bf16* __restrict__ qc)
{
    const int n = *n_sel;
    const int vecs = row_elems / 8;
    for (int row = blockIdx.x; row < n + kBM; row += gridDim.x) {
        uint4* dst = reinterpret_cast<uint4*>(qc + static_cast<int64_t>(row) * row_elems);
        if (row < n) {
            const int b = seq_of_row(cu_q, B, row);
            const uint4* src =
                reinterpret_cast<const uint4*>(q + (static_cast<int64_t>(b) * T + pos[row]) * row_elems);
            for (int v = threadIdx.x; v < vecs; v += blockDim.x) dst[v] = src[v];
        } else {
            for (int v = threadIdx.x; v < vecs; v += blockDim.x) dst[v] = make_uint4(0, 0, 0, 0);
        }
    }
}

}  // namespace logo
