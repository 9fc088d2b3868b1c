// colsum.cuh -- column sums of the per-block partial gradients that the
// gate, combine and transform backwards write ([nrows][ncols] fp32, one row
// per block of the producing kernel).
//
// A block of 1024 threads owns 32 columns: warp g adds rows g, g+32, g+64, ...
// of its lane's column in increasing order, then lane c of warp 0 adds the 32
// warp sums in warp order.  The order is fixed by the code, so the result is
// deterministic, and 32 rows in flight per column keep HBM busy where one
// thread per column walking every row was bound by load latency.
#pragma once

#include <cstdint>

namespace logo {
namespace {  // one copy per translation unit that launches it

constexpr int kColSumThreads = 1024;

// Columns [0, split) go to out0[c], columns [split, ncols) to out1[c - split];
// a null output skips its columns.
__global__ void __launch_bounds__(kColSumThreads) colsum_kernel(const float* __restrict__ part, int nrows,
                                                                int ncols, int split, float* __restrict__ out0,
                                                                float* __restrict__ out1)
{
    __shared__ float sh[32][33];
    const int lane = threadIdx.x & 31, g = threadIdx.x >> 5;
    const int col = blockIdx.x * 32 + lane;
    float s = 0.f;
    if (col < ncols) {
#pragma unroll 4
        for (int r = g; r < nrows; r += 32) s += part[static_cast<int64_t>(r) * ncols + col];
    }
    sh[g][lane] = s;
    __syncthreads();
    if (g == 0 && col < ncols) {
        float t = 0.f;
#pragma unroll
        for (int k = 0; k < 32; ++k) t += sh[k][lane];
        float* dst = col < split ? out0 : out1;
        if (dst) dst[col < split ? col : col - split] = t;
    }
}

inline int colsum_blocks(int ncols) { return (ncols + 31) / 32; }

}  // namespace
}  // namespace logo
