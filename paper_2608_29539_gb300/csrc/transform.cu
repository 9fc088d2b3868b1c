// transform.cu -- logo_branch_transform / _bwd: the per-head branch transforms
// of Eq. 5 that turn the local branch's Q/K/V into the global branch's,
//   LP: U^G_h = U^L_h A_h   (A_h a d x d matrix per head; the paper's default)
//   SO: U^G_h = U^L_h * s_h + b_h
// on either every row of a [B, T, H, d] tensor (K and V) or only the packed
// selected rows (Q: the global branch reads Q^G on those rows alone, so the
// transform of the other B*T - N rows is never computed).
//
// LP is a contraction of 2 d^2 FLOP per row and head against 4 d bytes moved:
// at d = 128 that is 64 FLOP/byte, more than the CUDA cores can keep up with
// at HBM speed, so it runs on the tensor cores.  On every row (K, V) a tcgen05
// pipeline: TMA brings 128-row tiles of one head into shared memory next to
// that head's A_h, one thread issues the MMAs into two TMEM buffers, four warps
// drain them.  On the packed selected rows (Q; rows gathered by position)
// warp-level mma.sync over 64-row tiles.  A block keeps one head's A_h and
// walks a strided share of its row tiles.  The backward computes
// dU^L = dU^G A_h^T on the same tiles and accumulates dA_h = U^L^T dU^G; per-
// block partial dA are reduced in block order by a second kernel
// (deterministic).  SO is elementwise; its per-block ds, db are summed by the
// fixed-order column sum of colsum.cuh (deterministic too).
#include <cuda_bf16.h>

#include <cstdint>

#include "colsum.cuh"
#include "attn_common.cuh"
#include "host_common.h"
#include "sm100.cuh"

namespace logo {
namespace {

constexpr int kTileRows = 64;
constexpr int kChunksPerHead = 16;  // blocks per head (row tiles strided among them)

// Row r of the listed set -> token index b*T + t (all rows: r itself).
struct RowSet {
    const int32_t* pos;    // packed positions, or NULL for every row
    const int32_t* cu_q;
    const int32_t* n_sel;  // device count of packed rows
    int B, T;
};

__device__ __forceinline__ int row_count(const RowSet& R)
{
    return R.pos ? *R.n_sel : R.B * R.T;
}

__device__ __forceinline__ int64_t row_token(const RowSet& R, int r)
{
    if (!R.pos) return r;
    const int b = seq_of_row(R.cu_q, R.B, r);
    return static_cast<int64_t>(b) * R.T + R.pos[r];
}

// [rows][D] bf16 tile in shared memory, 16-byte chunk c of row r stored at
// chunk c ^ (r & 7): the 8 rows an ldmatrix reads hit 8 different bank groups.
template <int D>
__device__ __forceinline__ uint32_t toff(int row, int chunk)
{
    return static_cast<uint32_t>(row * (D * 2) + ((chunk ^ (row & 7)) << 4));
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;\n" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_one() { asm volatile("cp.async.wait_group 1;\n" ::: "memory"); }

__device__ __forceinline__ void st_shared_b32(uint32_t addr, uint32_t v)
{
    asm volatile("st.shared.b32 [%0], %1;\n" ::"r"(addr), "r"(v) : "memory");
}

// Start the copies of rows [0, nrows) of a tile (token indices in tok[]) of
// head h into shared memory; rows past the end are zeroed with plain stores.
// The copies complete at the caller's cp.async wait.
template <int D>
__device__ __forceinline__ void load_tile_async(uint32_t dst, const logo_bf16* src, const int64_t* tok, int nrows,
                                                int H, int h, int nthreads)
{
    constexpr int kChunks = D / 8;
    for (int idx = threadIdx.x; idx < kTileRows * kChunks; idx += nthreads) {
        const int r = idx / kChunks, c = idx % kChunks;
        if (r < nrows) cp_async16(dst + toff<D>(r, c), src + (tok[r] * H + h) * D + c * 8);
        else st_shared_v4(dst + toff<D>(r, c), 0u, 0u, 0u, 0u);
    }
}

template <int D>
__device__ __forceinline__ void load_matrix_async(uint32_t dst, const logo_bf16* a, int nthreads)
{
    constexpr int kChunks = D / 8;
    for (int idx = threadIdx.x; idx < D * kChunks; idx += nthreads) {
        const int r = idx / kChunks, c = idx % kChunks;
        cp_async16(dst + toff<D>(r, c), a + r * D + c * 8);
    }
}

// token index of row r of the listed set, 0 past the end
__device__ __forceinline__ int64_t tile_token(const RowSet& R, int n, int r) { return r < n ? row_token(R, r) : 0; }

// LP forward: u_g[row] = u_l[row] A_h.  4 warps, 16 rows of the 64-row tile
// each.  A block walks a strided share of its head's row tiles with two tile
// buffers: the copies of A_h start before the row count is read, the token
// lists of the first two tiles are looked up together, and tile k+2 is
// fetched (cp.async) while tile k+1 is in flight and tile k is multiplied.
// A warp writes its results back over its own 16 rows of the tile (the only
// rows its MMAs read), so the stores to global memory leave as whole 2D-byte
// row pieces, two rows per warp instruction, instead of 16-byte fragments.
template <int D>
__global__ void __launch_bounds__(128) lp_fwd_kernel(const logo_bf16* __restrict__ u_l,
                                                     const logo_bf16* __restrict__ a, RowSet R, int H,
                                                     logo_bf16* __restrict__ u_g)
{
    constexpr int kTileBytes = kTileRows * D * 2;
    constexpr int kChunks = D / 8;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int64_t tok[2][kTileRows];
    const uint32_t sA = smem_u32(smem), sU = sA + D * D * 2;
    const int h = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mi = lane >> 3, rr = lane & 7, gid = lane >> 2, tig = lane & 3;
    load_matrix_async<D>(sA, a + static_cast<int64_t>(h) * D * D, 128);  // joins the first tile's group
    const int n = row_count(R);
    const int ntiles = (n + kTileRows - 1) / kTileRows;
    const int step = gridDim.x;
    int tile = blockIdx.x;
    if (tile >= ntiles) {  // no tile: let A_h's copies land before the block exits
        cp_async_wait_all();
        return;
    }
    {  // threads 0..63: rows of the first tile, 64..127: rows of the second
        const int which = threadIdx.x / kTileRows, r = threadIdx.x % kTileRows;
        tok[which][r] = tile_token(R, n, (tile + which * step) * kTileRows + r);
    }
    __syncthreads();
    load_tile_async<D>(sU, u_l, tok[0], min(kTileRows, n - tile * kTileRows), H, h, 128);
    cp_async_commit();
    if (tile + step < ntiles) {
        load_tile_async<D>(sU + kTileBytes, u_l, tok[1], min(kTileRows, n - (tile + step) * kTileRows), H, h, 128);
        cp_async_commit();
    }
    for (int k = 0; tile < ntiles; tile += step, ++k) {
        const int buf = k & 1;
        const int nr = min(kTileRows, n - tile * kTileRows);
        if (tile + step < ntiles) cp_async_wait_one();  // tile k+1 may stay in flight
        else cp_async_wait_all();
        __syncthreads();
        const uint32_t sT = sU + buf * kTileBytes;
        float acc[D / 8][4];
#pragma unroll
        for (int nt = 0; nt < D / 8; ++nt)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;
#pragma unroll
        for (int ks = 0; ks < D / 16; ++ks) {
            uint32_t fa[4];
            ldsm_x4(sT + toff<D>(warp * 16 + (mi & 1) * 8 + rr, 2 * ks + (mi >> 1)), fa[0], fa[1], fa[2], fa[3]);
#pragma unroll
            for (int np = 0; np < D / 16; ++np) {
                uint32_t b0, b1, b2, b3;  // A_h rows k (input dim), columns n (output dim)
                ldsm_x4_trans(sA + toff<D>(16 * ks + (mi & 1) * 8 + rr, 2 * np + (mi >> 1)), b0, b1, b2, b3);
                mma_bf16_16816(acc[2 * np], fa, b0, b1);
                mma_bf16_16816(acc[2 * np + 1], fa, b2, b3);
            }
        }
        __syncwarp();
#pragma unroll
        for (int half = 0; half < 2; ++half) {
            const int r = warp * 16 + gid + half * 8;
#pragma unroll
            for (int nt = 0; nt < D / 8; ++nt)
                st_shared_b32(sT + toff<D>(r, nt) + 4 * tig, pack_bf16x2(acc[nt][2 * half], acc[nt][2 * half + 1]));
        }
        __syncwarp();
#pragma unroll
        for (int idx = lane; idx < 16 * kChunks; idx += 32) {
            const int r = warp * 16 + idx / kChunks, c = idx % kChunks;
            if (r < nr) {
                const uint4 v = ld_shared_v4(sT + toff<D>(r, c));
                *reinterpret_cast<uint4*>(u_g + (tok[buf][r] * H + h) * D + c * 8) = v;
            }
        }
        __syncthreads();  // buffer buf and tok[buf] are free
        const int after = tile + 2 * step;  // tile k+2 goes where tile k was
        if (after < ntiles) {
            if (threadIdx.x < kTileRows) tok[buf][threadIdx.x] = tile_token(R, n, after * kTileRows + threadIdx.x);
            __syncthreads();
            load_tile_async<D>(sT, u_l, tok[buf], min(kTileRows, n - after * kTileRows), H, h, 128);
            cp_async_commit();
        }
    }
}

// LP backward: du_l[row] (+)= du_g[row] A_h^T, and dA_h += u_l^T du_g over the
// block's rows.  D/16 warps: for dU, warp w takes rows 16 (w % 4).. and output
// columns 64 (w / 4)..; for dA, rows 16w.. of the D x D result.
// part: [H][gridDim.x][D][D] float32.
template <int D>
__global__ void __launch_bounds__(D * 2) lp_bwd_kernel(const logo_bf16* __restrict__ u_l,
                                                       const logo_bf16* __restrict__ a,
                                                       const logo_bf16* __restrict__ du_g, RowSet R, int H,
                                                       logo_bf16* __restrict__ du_l, int accumulate,
                                                       float* __restrict__ part)
{
    constexpr int kThreads = D * 2;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int64_t tok[kTileRows];
    const uint32_t sA = smem_u32(smem), sU = sA + D * D * 2, sG = sU + kTileRows * D * 2;
    const int h = blockIdx.y, warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int mi = lane >> 3, rr = lane & 7, gid = lane >> 2, tig = lane & 3;
    load_matrix_async<D>(sA, a + static_cast<int64_t>(h) * D * D, kThreads);  // lands with the first tile
    float acc_a[D / 8][4];
#pragma unroll
    for (int nt = 0; nt < D / 8; ++nt)
#pragma unroll
        for (int i = 0; i < 4; ++i) acc_a[nt][i] = 0.f;
    const int n = row_count(R);
    const int ntiles = (n + kTileRows - 1) / kTileRows;
    const int rg = warp & 3, cb = (warp >> 2) * 64;  // dU: row group and first output column
    for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
        const int r0 = tile * kTileRows, nr = min(kTileRows, n - r0);
        if (threadIdx.x < kTileRows) tok[threadIdx.x] = threadIdx.x < nr ? row_token(R, r0 + threadIdx.x) : 0;
        __syncthreads();
        load_tile_async<D>(sU, u_l, tok, nr, H, h, kThreads);
        load_tile_async<D>(sG, du_g, tok, nr, H, h, kThreads);
        cp_async_commit();
        cp_async_wait_all();
        __syncthreads();
        // dU = dG A^T: rows 16 rg.., output columns cb .. cb + 63 (A_h rows i)
        {
            float acc[8][4];
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[nt][i] = 0.f;
#pragma unroll
            for (int ks = 0; ks < D / 16; ++ks) {  // k: A_h columns j
                uint32_t fa[4];
                ldsm_x4(sG + toff<D>(rg * 16 + (mi & 1) * 8 + rr, 2 * ks + (mi >> 1)), fa[0], fa[1], fa[2], fa[3]);
#pragma unroll
                for (int np = 0; np < 4; ++np) {
                    uint32_t b0, b1, b2, b3;  // B(k = j, n = i) = A_h[i][j]: rows n, k contiguous
                    ldsm_x4(sA + toff<D>(cb + np * 16 + (mi >> 1) * 8 + rr, 2 * ks + (mi & 1)), b0, b1, b2, b3);
                    mma_bf16_16816(acc[2 * np], fa, b0, b1);
                    mma_bf16_16816(acc[2 * np + 1], fa, b2, b3);
                }
            }
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                const int r = rg * 16 + gid + half * 8;
                if (r < nr) {
                    logo_bf16* dst = du_l + (tok[r] * H + h) * D + cb + 2 * tig;
#pragma unroll
                    for (int nt = 0; nt < 8; ++nt) {
                        float x0 = acc[nt][2 * half], x1 = acc[nt][2 * half + 1];
                        uint32_t* p = reinterpret_cast<uint32_t*>(dst + nt * 8);
                        if (accumulate) {
                            const float2 old = __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
                            x0 += old.x;
                            x1 += old.y;
                        }
                        *p = pack_bf16x2(x0, x1);
                    }
                }
            }
        }
        // dA += U^T dG: result rows i = 16 warp .., all columns j; k = the tile's rows
#pragma unroll
        for (int ks = 0; ks < kTileRows / 16; ++ks) {
            uint32_t fa[4];  // A(m = i, k = r) = U[r][i]: stored rows k, m contiguous
            ldsm_x4_trans(sU + toff<D>(16 * ks + (mi >> 1) * 8 + rr, 2 * warp + (mi & 1)), fa[0], fa[1], fa[2], fa[3]);
#pragma unroll
            for (int np = 0; np < D / 16; ++np) {
                uint32_t b0, b1, b2, b3;  // B(k = r, n = j) = dG[r][j]
                ldsm_x4_trans(sG + toff<D>(16 * ks + (mi & 1) * 8 + rr, 2 * np + (mi >> 1)), b0, b1, b2, b3);
                mma_bf16_16816(acc_a[2 * np], fa, b0, b1);
                mma_bf16_16816(acc_a[2 * np + 1], fa, b2, b3);
            }
        }
        __syncthreads();
    }
    cp_async_wait_all();  // a block with no tile still has A_h's copies in flight
    float* pp = part + (static_cast<int64_t>(h) * gridDim.x + blockIdx.x) * D * D;
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const int i = warp * 16 + gid + half * 8;
#pragma unroll
        for (int nt = 0; nt < D / 8; ++nt) {
            pp[i * D + nt * 8 + 2 * tig] = acc_a[nt][2 * half];
            pp[i * D + nt * 8 + 2 * tig + 1] = acc_a[nt][2 * half + 1];
        }
    }
}

// out[h][e] = sum over c (in order) of part[h][c][e], e < per_head.
__global__ void __launch_bounds__(256) reduce_parts_kernel(const float* __restrict__ part, int nchunk, int per_head,
                                                           int H, float* __restrict__ out)
{
    const int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (e >= static_cast<int64_t>(H) * per_head) return;
    const int h = static_cast<int>(e / per_head), x = static_cast<int>(e % per_head);
    float s = 0.f;
    for (int c = 0; c < nchunk; ++c) s += part[(static_cast<int64_t>(h) * nchunk + c) * per_head + x];
    out[e] = s;
}

// SO forward: u_g = u_l * s + b on the listed rows; a thread per 8-element vector.
__global__ void __launch_bounds__(256) so_fwd_kernel(const logo_bf16* __restrict__ u_l, const float* __restrict__ s,
                                                     const float* __restrict__ b, RowSet R, int H, int D,
                                                     logo_bf16* __restrict__ u_g)
{
    const int nvec = H * D / 8;
    const int64_t total = static_cast<int64_t>(row_count(R)) * nvec;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int r = static_cast<int>(i / nvec), v = static_cast<int>(i % nvec);
        const int64_t off = row_token(R, r) * H * D + v * 8;
        const uint4 raw = *reinterpret_cast<const uint4*>(u_l + off);
        const __nv_bfloat162* x = reinterpret_cast<const __nv_bfloat162*>(&raw);
        uint4 o;
        uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float2 f = __bfloat1622float2(x[q]);
            const int e = v * 8 + 2 * q;
            ow[q] = pack_bf16x2(fmaf(f.x, s[e], b[e]), fmaf(f.y, s[e + 1], b[e + 1]));
        }
        *reinterpret_cast<uint4*>(u_g + off) = o;
    }
}

// SO backward: du_l (+)= du_g * s; ds += du_g * u_l, db += du_g.  A thread owns
// fixed vectors (VPT of them) of the [H, D] row for all rows of its block.
// part: [gridDim.x][2][H*D] float32 (ds, db).
template <int VPT>
__global__ void __launch_bounds__(256) so_bwd_kernel(const logo_bf16* __restrict__ u_l, const float* __restrict__ s,
                                                     const logo_bf16* __restrict__ du_g, RowSet R, int H, int D,
                                                     logo_bf16* __restrict__ du_l, int accumulate,
                                                     float* __restrict__ part)
{
    const int nvec = H * D / 8;
    float acc_s[VPT][8], acc_b[VPT][8];
#pragma unroll
    for (int k = 0; k < VPT; ++k)
#pragma unroll
        for (int i = 0; i < 8; ++i) acc_s[k][i] = acc_b[k][i] = 0.f;
    const int n = row_count(R);
    for (int r = blockIdx.x; r < n; r += gridDim.x) {
        const int64_t base = row_token(R, r) * H * D;
#pragma unroll
        for (int k = 0; k < VPT; ++k) {
            const int v = threadIdx.x + k * 256;
            if (v >= nvec) continue;
            const uint4 gu = *reinterpret_cast<const uint4*>(du_g + base + v * 8);
            const uint4 uu = *reinterpret_cast<const uint4*>(u_l + base + v * 8);
            const __nv_bfloat162* g2 = reinterpret_cast<const __nv_bfloat162*>(&gu);
            const __nv_bfloat162* u2 = reinterpret_cast<const __nv_bfloat162*>(&uu);
            uint4 prev = make_uint4(0u, 0u, 0u, 0u);
            if (accumulate) prev = *reinterpret_cast<const uint4*>(du_l + base + v * 8);
            const __nv_bfloat162* p2 = reinterpret_cast<const __nv_bfloat162*>(&prev);
            uint4 o;
            uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float2 g = __bfloat1622float2(g2[q]), u = __bfloat1622float2(u2[q]);
                const int e = v * 8 + 2 * q;
                float x0 = g.x * s[e], x1 = g.y * s[e + 1];
                if (accumulate) {
                    const float2 pv = __bfloat1622float2(p2[q]);
                    x0 += pv.x;
                    x1 += pv.y;
                }
                ow[q] = pack_bf16x2(x0, x1);
                acc_s[k][2 * q] = fmaf(g.x, u.x, acc_s[k][2 * q]);
                acc_s[k][2 * q + 1] = fmaf(g.y, u.y, acc_s[k][2 * q + 1]);
                acc_b[k][2 * q] += g.x;
                acc_b[k][2 * q + 1] += g.y;
            }
            *reinterpret_cast<uint4*>(du_l + base + v * 8) = o;
        }
    }
    const int64_t hd = static_cast<int64_t>(H) * D;
#pragma unroll
    for (int k = 0; k < VPT; ++k) {
        const int v = threadIdx.x + k * 256;
        if (v >= nvec) continue;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            part[static_cast<int64_t>(blockIdx.x) * 2 * hd + v * 8 + i] = acc_s[k][i];
            part[static_cast<int64_t>(blockIdx.x) * 2 * hd + hd + v * 8 + i] = acc_b[k][i];
        }
    }
}

// ------------------------------------------------------------------------
// LP on every row (K and V) with tcgen05: a tile is 128 rows of one head.
// Roles: warp 0 TMA (A_h once, U tiles through a 2-deep ring), warp 1 MMA
// issuer (D[128 x D] = U_tile A_h into one of two TMEM buffers), warps 2..5
// epilogue (TMEM -> bf16 -> global).  A CTA keeps one head; the row tiles of
// that head are strided over gridDim.x CTAs.  Shared memory: A_h as 64-column
// halves of [D rows][64] (128-byte swizzle), read as the MN-major B operand;
// U tiles as 64-column halves of [128 rows][64], the K-major A operand.
struct LpTcParams {
    CUtensorMap tm_u;   // u_l [B,T,H,D] as (d, h, t, b), box {64, 1, 128, 1}
    CUtensorMap tm_a;   // a [H*D rows][D] as (j, 1, row, 1), box {64, 1, D, 1}
    logo_bf16* u_g;
    int B, T, H;
};

template <int D>
struct LpTcCfg {
    static constexpr int kHalfA = D * 128;                 // [D rows][64] bf16
    static constexpr int kABytes = (D / 64) * kHalfA;
    static constexpr int kHalfU = 128 * 128;               // [128 rows][64] bf16
    static constexpr int kUBytes = (D / 64) * kHalfU;
    static constexpr int kOffA = 0;
    static constexpr int kOffU = kABytes;                  // 2 stages
    static constexpr int kSmemBytes = kOffU + 2 * kUBytes + 1024;
    static constexpr uint32_t kTmemCols = D == 128 ? 256 : 128;  // two D-column result buffers
};

template <int D>
__global__ void __launch_bounds__(192, 1) lp_tc_fwd_kernel(const __grid_constant__ LpTcParams p)
{
    using C = LpTcCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_a, bar_u_full[2], bar_u_empty[2], bar_t_full[2], bar_t_empty[2], bar_drain;
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.y;
    const int tiles_per_seq = (p.T + 127) / 128;
    const int ntiles = p.B * tiles_per_seq;
    const uint32_t sA = smem_u32(smem + C::kOffA), sU = smem_u32(smem + C::kOffU);
    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_a), 1);
        mbar_init(smem_u32(&bar_drain), 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bar_u_full[s]), 1);
            mbar_init(smem_u32(&bar_u_empty[s]), 1);
            mbar_init(smem_u32(&bar_t_full[s]), 1);
            mbar_init(smem_u32(&bar_t_empty[s]), 128);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_sh), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_desc(&p.tm_u);
            tma_prefetch_desc(&p.tm_a);
            const uint64_t pol_u = policy_evict_first(), pol_a = policy_evict_last();
            mbar_arrive_expect_tx(smem_u32(&bar_a), C::kABytes);
            for (int s = 0; s < D / 64; ++s)
                tma_load_4d(sA + s * C::kHalfA, &p.tm_a, smem_u32(&bar_a), 64 * s, 0, h * D, 0, pol_a);
            int k = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++k) {
                const int st = k & 1;
                if (!(ok = mbar_wait(smem_u32(&bar_u_empty[st]), ((k >> 1) & 1) ^ 1, &abort_flag))) break;
                const int b = tile / tiles_per_seq, t0 = (tile % tiles_per_seq) * 128;
                mbar_arrive_expect_tx(smem_u32(&bar_u_full[st]), C::kUBytes);
                for (int s = 0; s < D / 64; ++s)
                    tma_load_4d(sU + st * C::kUBytes + s * C::kHalfU, &p.tm_u, smem_u32(&bar_u_full[st]), 64 * s, h,
                                t0, b, pol_u);
            }
            if (!ok) {  // let the copies already issued land before the CTA exits
                mbar_wait_drain(smem_u32(&bar_a), 0);
                for (int j = k - 2 > 0 ? k - 2 : 0; j < k; ++j)
                    mbar_wait_drain(smem_u32(&bar_u_full[j & 1]), (j >> 1) & 1);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(128, D, false, true);
            bool ok = mbar_wait(smem_u32(&bar_a), 0, &abort_flag);
            int k = 0;
            for (int tile = blockIdx.x; ok && tile < ntiles; tile += gridDim.x, ++k) {
                const int st = k & 1;
                if (!(ok = mbar_wait(smem_u32(&bar_u_full[st]), (k >> 1) & 1, &abort_flag))) break;
                if (!(ok = mbar_wait(smem_u32(&bar_t_empty[st]), ((k >> 1) & 1) ^ 1, &abort_flag))) break;
                tc_fence_after();
                const uint32_t ub = sU + st * C::kUBytes;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {
                    const uint32_t ka = (ks >> 2) * C::kHalfU + (ks & 3) * 32;  // U: K-major halves of 64
                    umma_bf16_ss(tmem + st * D, sdesc_sw128(ub + ka, 16, 1024),
                                 sdesc_sw128(sA + ks * 2048, C::kHalfA, 1024), idesc, ks > 0 ? 1u : 0u);
                }
                umma_commit(smem_u32(&bar_u_empty[st]));
                umma_commit(smem_u32(&bar_t_full[st]));
            }
            if (!ok) {
                umma_commit(smem_u32(&bar_drain));
                mbar_wait_drain(smem_u32(&bar_drain), 0);
            }
        }
    } else {
        // epilogue: warp w reads TMEM lanes 32 (w % 4) .. (its rows of the tile)
        const int quad = warp & 3;
        const int r = quad * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        int k = 0;
        for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++k) {
            const int st = k & 1;
            const bool ok = mbar_wait(smem_u32(&bar_t_full[st]), (k >> 1) & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
            const int b = tile / tiles_per_seq, t = (tile % tiles_per_seq) * 128 + r;
            logo_bf16* dst = p.u_g + ((static_cast<int64_t>(b) * p.T + t) * p.H + h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_off + st * D + c * 32, v);
                tmem_wait_ld();
                if (c == D / 32 - 1) {
                    tc_fence_before();
                    mbar_arrive(smem_u32(&bar_t_empty[st]));
                }
                if (t < p.T) {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(v[8 * q4 + 0]), __uint_as_float(v[8 * q4 + 1]));
                        w.y = pack_bf16x2(__uint_as_float(v[8 * q4 + 2]), __uint_as_float(v[8 * q4 + 3]));
                        w.z = pack_bf16x2(__uint_as_float(v[8 * q4 + 4]), __uint_as_float(v[8 * q4 + 5]));
                        w.w = pack_bf16x2(__uint_as_float(v[8 * q4 + 6]), __uint_as_float(v[8 * q4 + 7]));
                        *reinterpret_cast<uint4*>(dst + c * 32 + q4 * 8) = w;
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

template <int D>
int launch_lp_tc_fwd(const logo_bf16* u_l, const logo_bf16* a, const logo_dims& d, logo_bf16* u_g, cudaStream_t st)
{
    LpTcParams prm{};
    if (!encode_bf16_4d(&prm.tm_u, u_l, D, d.Hq, d.T, d.B, 64, 128) ||
        !encode_bf16_4d(&prm.tm_a, a, D, 1, static_cast<uint64_t>(d.Hq) * D, 1, 64, D))
        return LOGO_ERR_CUDA;
    prm.u_g = u_g;
    prm.B = d.B;
    prm.T = d.T;
    prm.H = d.Hq;
    if (set_smem_limit(lp_tc_fwd_kernel<D>, LpTcCfg<D>::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
    const int ntiles = d.B * ((d.T + 127) / 128);
    int per_head = (2 * device_sm_count()) / d.Hq;
    per_head = per_head < 1 ? 1 : (per_head > ntiles ? ntiles : per_head);
    lp_tc_fwd_kernel<D><<<dim3(per_head, d.Hq), 192, LpTcCfg<D>::kSmemBytes, st>>>(prm);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

// LP backward on every row, d = 128, with tcgen05.  Per 128-row tile of one
// head: dU = dG A_h^T (A_h read as the K-major B operand: its rows are the
// output dimension i, its columns the contracted j) into one of two TMEM
// buffers, drained to du_l by warps 2..5; and dA_h += U^T dG (both tiles read
// as MN-major operands: rows are the contracted dimension) accumulated in TMEM
// over all the CTA's tiles, written as the CTA's partial at the end.
struct LpTcBwdParams {
    CUtensorMap tm_u, tm_g, tm_a;
    logo_bf16* du_l;
    float* part;  // [H][gridDim.x][D][D]
    int B, T, H, accumulate;
};

struct LpTcBwdCfg {
    static constexpr int D = 128;
    static constexpr int kHalf = 128 * 128;          // [128 rows][64] bf16
    static constexpr int kTile = 2 * kHalf;          // 128 rows x 128
    static constexpr int kOffA = 0;
    static constexpr int kOffU = kTile;              // 2 stages of (U, G)
    static constexpr int kSmemBytes = kOffU + 4 * kTile + 1024;
    static constexpr uint32_t kColDA = 256;          // dU buffers at 0 and 128
    static constexpr uint32_t kTmemCols = 512;
};

__global__ void __launch_bounds__(192, 1) lp_tc_bwd_kernel(const __grid_constant__ LpTcBwdParams p)
{
    using C = LpTcBwdCfg;
    constexpr int D = C::D;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_a, bar_in_full[2], bar_in_empty[2], bar_t_full[2], bar_t_empty[2];
    __shared__ __align__(8) uint64_t bar_da, bar_drain;
    __shared__ uint32_t tmem_sh;
    __shared__ volatile int abort_flag;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = blockIdx.y;
    const int tiles_per_seq = (p.T + 127) / 128;
    const int ntiles = p.B * tiles_per_seq;
    const uint32_t sA = smem_u32(smem + C::kOffA), sIn = smem_u32(smem + C::kOffU);
    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_a), 1);
        mbar_init(smem_u32(&bar_da), 1);
        mbar_init(smem_u32(&bar_drain), 1);
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bar_in_full[s]), 1);
            mbar_init(smem_u32(&bar_in_empty[s]), 1);
            mbar_init(smem_u32(&bar_t_full[s]), 1);
            mbar_init(smem_u32(&bar_t_empty[s]), 128);
        }
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(&tmem_sh), C::kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    if (warp == 0) {
        if (lane == 0) {
            tma_prefetch_desc(&p.tm_u);
            tma_prefetch_desc(&p.tm_g);
            tma_prefetch_desc(&p.tm_a);
            const uint64_t pol = policy_evict_first(), pol_a = policy_evict_last();
            mbar_arrive_expect_tx(smem_u32(&bar_a), C::kTile);
            for (int s = 0; s < 2; ++s) tma_load_4d(sA + s * C::kHalf, &p.tm_a, smem_u32(&bar_a), 64 * s, 0, h * D, 0, pol_a);
            int k = 0;
            bool ok = true;
            for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++k) {
                const int st = k & 1;
                if (!(ok = mbar_wait(smem_u32(&bar_in_empty[st]), ((k >> 1) & 1) ^ 1, &abort_flag))) break;
                const int b = tile / tiles_per_seq, t0 = (tile % tiles_per_seq) * 128;
                const uint32_t bar = smem_u32(&bar_in_full[st]);
                const uint32_t ub = sIn + st * 2 * C::kTile, gb = ub + C::kTile;
                mbar_arrive_expect_tx(bar, 2 * C::kTile);
                for (int s = 0; s < 2; ++s) {
                    tma_load_4d(ub + s * C::kHalf, &p.tm_u, bar, 64 * s, h, t0, b, pol);
                    tma_load_4d(gb + s * C::kHalf, &p.tm_g, bar, 64 * s, h, t0, b, pol);
                }
            }
            if (!ok) {
                mbar_wait_drain(smem_u32(&bar_a), 0);
                for (int j = k - 2 > 0 ? k - 2 : 0; j < k; ++j)
                    mbar_wait_drain(smem_u32(&bar_in_full[j & 1]), (j >> 1) & 1);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            constexpr uint32_t id_du = idesc_bf16_f32(128, D, false, false);  // G K-major x A_h K-major
            constexpr uint32_t id_da = idesc_bf16_f32(D, D, true, true);      // U^T, G: both MN-major
            bool ok = mbar_wait(smem_u32(&bar_a), 0, &abort_flag);
            int k = 0;
            for (int tile = blockIdx.x; ok && tile < ntiles; tile += gridDim.x, ++k) {
                const int st = k & 1;
                if (!(ok = mbar_wait(smem_u32(&bar_in_full[st]), (k >> 1) & 1, &abort_flag))) break;
                if (!(ok = mbar_wait(smem_u32(&bar_t_empty[st]), ((k >> 1) & 1) ^ 1, &abort_flag))) break;
                tc_fence_after();
                const uint32_t ub = sIn + st * 2 * C::kTile, gb = ub + C::kTile;
#pragma unroll
                for (int ks = 0; ks < D / 16; ++ks) {  // contracted: j
                    const uint32_t off = (ks >> 2) * C::kHalf + (ks & 3) * 32;
                    umma_bf16_ss(tmem + st * D, sdesc_sw128(gb + off, 16, 1024), sdesc_sw128(sA + off, 16, 1024), id_du,
                                 ks > 0 ? 1u : 0u);
                }
#pragma unroll
                for (int ks = 0; ks < 128 / 16; ++ks) {  // contracted: the tile's rows
                    umma_bf16_ss(tmem + C::kColDA, sdesc_sw128(ub + ks * 2048, C::kHalf, 1024),
                                 sdesc_sw128(gb + ks * 2048, C::kHalf, 1024), id_da, (k > 0 || ks > 0) ? 1u : 0u);
                }
                umma_commit(smem_u32(&bar_in_empty[st]));
                umma_commit(smem_u32(&bar_t_full[st]));
            }
            // dA complete (every MMA of this thread before the commit); also on a
            // CTA with no tile, so that the epilogue's final wait ends
            if (ok) umma_commit(smem_u32(&bar_da));
            if (!ok) {
                umma_commit(smem_u32(&bar_drain));
                mbar_wait_drain(smem_u32(&bar_drain), 0);
            }
        }
    } else {
        const int quad = warp & 3;
        const int r = quad * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        int k = 0;
        bool ok = true;
        for (int tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++k) {
            const int st = k & 1;
            ok = mbar_wait(smem_u32(&bar_t_full[st]), (k >> 1) & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
            const int b = tile / tiles_per_seq, t = (tile % tiles_per_seq) * 128 + r;
            logo_bf16* dst = p.du_l + ((static_cast<int64_t>(b) * p.T + t) * p.H + h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_off + st * D + c * 32, v);
                tmem_wait_ld();
                if (c == D / 32 - 1) {
                    tc_fence_before();
                    mbar_arrive(smem_u32(&bar_t_empty[st]));
                }
                if (t < p.T) {
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
                        float x[8];
#pragma unroll
                        for (int e = 0; e < 8; ++e) x[e] = __uint_as_float(v[8 * q4 + e]);
                        uint4* dp = reinterpret_cast<uint4*>(dst + c * 32 + q4 * 8);
                        if (p.accumulate) {
                            const uint4 old = *dp;
                            const __nv_bfloat162* o2 = reinterpret_cast<const __nv_bfloat162*>(&old);
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const float2 f = __bfloat1622float2(o2[e]);
                                x[2 * e] += f.x;
                                x[2 * e + 1] += f.y;
                            }
                        }
                        uint4 w;
                        w.x = pack_bf16x2(x[0], x[1]);
                        w.y = pack_bf16x2(x[2], x[3]);
                        w.z = pack_bf16x2(x[4], x[5]);
                        w.w = pack_bf16x2(x[6], x[7]);
                        *dp = w;
                    }
                }
            }
        }
        // the CTA's dA partial: lane r holds row i = r, columns j
        float* pp = p.part + ((static_cast<int64_t>(h) * gridDim.x + blockIdx.x) * D + r) * D;
        if (ok && k == 0) {  // no tile: a zero partial (the launch gives every CTA one)
            for (int j = 0; j < D; j += 4) *reinterpret_cast<float4*>(pp + j) = make_float4(0.f, 0.f, 0.f, 0.f);
        } else if (ok && mbar_wait(smem_u32(&bar_da), 0, &abort_flag)) {
            tc_fence_after();
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t v[32];
                tmem_ld32(tmem + lane_off + C::kColDA + c * 32, v);
                tmem_wait_ld();
#pragma unroll
                for (int e = 0; e < 32; e += 4)
                    *reinterpret_cast<float4*>(pp + c * 32 + e) =
                        make_float4(__uint_as_float(v[e]), __uint_as_float(v[e + 1]), __uint_as_float(v[e + 2]),
                                    __uint_as_float(v[e + 3]));
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

int launch_lp_tc_bwd(const logo_bf16* u_l, const logo_bf16* a, const logo_bf16* du_g, const logo_dims& d,
                     logo_bf16* du_l, int accumulate, float* da, float* part, cudaStream_t st)
{
    constexpr int D = 128;
    LpTcBwdParams prm{};
    if (!encode_bf16_4d(&prm.tm_u, u_l, D, d.Hq, d.T, d.B, 64, 128) ||
        !encode_bf16_4d(&prm.tm_g, du_g, D, d.Hq, d.T, d.B, 64, 128) ||
        !encode_bf16_4d(&prm.tm_a, a, D, 1, static_cast<uint64_t>(d.Hq) * D, 1, 64, D))
        return LOGO_ERR_CUDA;
    prm.du_l = du_l;
    prm.part = part;
    prm.B = d.B;
    prm.T = d.T;
    prm.H = d.Hq;
    prm.accumulate = accumulate;
    if (set_smem_limit(lp_tc_bwd_kernel, LpTcBwdCfg::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
    const int ntiles = d.B * ((d.T + 127) / 128);
    int per_head = device_sm_count() / d.Hq;
    per_head = per_head < 1 ? 1 : (per_head > ntiles ? ntiles : per_head);
    per_head = per_head > kChunksPerHead ? kChunksPerHead : per_head;  // the workspace holds that many partials
    lp_tc_bwd_kernel<<<dim3(per_head, d.Hq), 192, LpTcBwdCfg::kSmemBytes, st>>>(prm);
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    const int64_t total = static_cast<int64_t>(d.Hq) * D * D;
    reduce_parts_kernel<<<static_cast<unsigned>((total + 255) / 256), 256, 0, st>>>(part, per_head, D * D, d.Hq, da);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

int so_vpt(const logo_dims& d)
{
    const int nvec = d.Hq * d.D / 8;
    const int need = (nvec + 255) / 256;
    return need <= 1 ? 1 : need <= 2 ? 2 : 4;
}

int so_bwd_blocks(const logo_dims& d)
{
    const int64_t rows = static_cast<int64_t>(d.B) * d.T;
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * 4;
    return static_cast<int>(rows < cap ? rows : cap);
}

int check_transform(const logo_dims& d, const void* u, const void* out)
{
    if (d.B < 1 || d.T < 1 || d.Hq < 1) return LOGO_ERR_INVALID_ARG;
    if (d.D != 64 && d.D != 128) return LOGO_ERR_UNSUPPORTED;
    if (static_cast<int64_t>(d.B) * d.T > (1ll << 30)) return LOGO_ERR_UNSUPPORTED;
    if (d.Hq * d.D > 8192) return LOGO_ERR_UNSUPPORTED;
    if (!aligned16(u) || !aligned16(out)) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

template <int D>
int launch_lp_fwd(const logo_bf16* u_l, const logo_bf16* a, const RowSet& R, int H, logo_bf16* u_g,
                  cudaStream_t st)
{
    const int smem = D * D * 2 + 2 * kTileRows * D * 2;  // A_h and two row tiles
    if (set_smem_limit(lp_fwd_kernel<D>, smem) != cudaSuccess) return LOGO_ERR_CUDA;
    // one wave: blocks per SM as shared memory allows (3 at d = 128, 64 KB each),
    // split evenly over the heads; each block walks a strided share of its head's tiles
    const int per_sm = D == 128 ? 3 : 6;
    int chunks = per_sm * device_sm_count() / H;
    chunks = chunks < 1 ? 1 : chunks > 64 ? 64 : chunks;
    lp_fwd_kernel<D><<<dim3(chunks, H), 128, smem, st>>>(u_l, a, R, H, u_g);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

template <int D>
int launch_lp_bwd(const logo_bf16* u_l, const logo_bf16* a, const logo_bf16* du_g, const RowSet& R, int H,
                  logo_bf16* du_l, int accumulate, float* da, float* part, cudaStream_t st)
{
    const int smem = D * D * 2 + 2 * kTileRows * D * 2;
    if (set_smem_limit(lp_bwd_kernel<D>, smem) != cudaSuccess) return LOGO_ERR_CUDA;
    lp_bwd_kernel<D><<<dim3(kChunksPerHead, H), D * 2, smem, st>>>(u_l, a, du_g, R, H, du_l, accumulate, part);
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    const int64_t total = static_cast<int64_t>(H) * D * D;
    reduce_parts_kernel<<<static_cast<unsigned>((total + 255) / 256), 256, 0, st>>>(part, kChunksPerHead, D * D, H,
                                                                                   da);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

}  // namespace
int transform_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" int logo_branch_transform(const logo_bf16* u_l, const logo_bf16* a_lp, const float* s_so,
                                     const float* b_so, const int32_t* pos, const int32_t* cu_q,
                                     const int32_t* n_sel_total, logo_bf16* u_g, logo_dims dims, void* stream)
{
    int rc = check_transform(dims, u_l, u_g);
    if (rc != LOGO_OK) return rc;
    if (!u_l || !u_g) return LOGO_ERR_INVALID_ARG;
    if ((a_lp != nullptr) == (s_so != nullptr || b_so != nullptr)) return LOGO_ERR_INVALID_ARG;  // exactly one form
    if (!a_lp && (!s_so || !b_so)) return LOGO_ERR_INVALID_ARG;
    if (pos && (!cu_q || !n_sel_total)) return LOGO_ERR_INVALID_ARG;
    if (a_lp && !aligned16(a_lp)) return LOGO_ERR_UNSUPPORTED;
    const RowSet R{pos, cu_q, n_sel_total, dims.B, dims.T};
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (a_lp && !pos) {  // every row: the tcgen05 pipeline
        return dims.D == 128 ? launch_lp_tc_fwd<128>(u_l, a_lp, dims, u_g, st)
                             : launch_lp_tc_fwd<64>(u_l, a_lp, dims, u_g, st);
    }
    if (a_lp) {  // the packed selected rows (Q): warp-level MMA over gathered rows
        return dims.D == 128 ? launch_lp_fwd<128>(u_l, a_lp, R, dims.Hq, u_g, st)
                             : launch_lp_fwd<64>(u_l, a_lp, R, dims.Hq, u_g, st);
    }
    const int64_t work = static_cast<int64_t>(dims.B) * dims.T * dims.Hq * dims.D / 8;
    const int64_t cap = static_cast<int64_t>(device_sm_count()) * 8;
    const int64_t blocks = (work + 255) / 256;
    so_fwd_kernel<<<static_cast<unsigned>(blocks < cap ? blocks : cap), 256, 0, st>>>(u_l, s_so, b_so, R, dims.Hq,
                                                                                       dims.D, u_g);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

extern "C" size_t logo_branch_transform_bwd_workspace_size(logo_dims dims)
{
    if (dims.B < 1 || dims.T < 1 || dims.Hq < 1 || (dims.D != 64 && dims.D != 128) || dims.Hq * dims.D > 8192)
        return 0;
    const size_t lp = static_cast<size_t>(dims.Hq) * kChunksPerHead * dims.D * dims.D * sizeof(float);
    const size_t so = static_cast<size_t>(so_bwd_blocks(dims)) * 2 * dims.Hq * dims.D * sizeof(float);
    return lp > so ? lp : so;
}

extern "C" int logo_branch_transform_bwd(const logo_bf16* u_l, const logo_bf16* a_lp, const float* s_so,
                                         const int32_t* pos, const int32_t* cu_q, const int32_t* n_sel_total,
                                         const logo_bf16* du_g, logo_bf16* du_l, int accumulate, float* da_lp,
                                         float* ds_so, float* db_so, logo_dims dims, void* workspace,
                                         size_t workspace_bytes, void* stream)
{
    int rc = check_transform(dims, u_l, du_l);
    if (rc != LOGO_OK) return rc;
    if (!u_l || !du_g || !du_l) return LOGO_ERR_INVALID_ARG;
    if ((a_lp != nullptr) == (s_so != nullptr)) return LOGO_ERR_INVALID_ARG;  // exactly one form
    if (a_lp && !da_lp) return LOGO_ERR_INVALID_ARG;
    if (accumulate != 0 && accumulate != 1) return LOGO_ERR_INVALID_ARG;
    if (pos && (!cu_q || !n_sel_total)) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(du_g) || (a_lp && !aligned16(a_lp))) return LOGO_ERR_UNSUPPORTED;
    if (!workspace || workspace_bytes < logo_branch_transform_bwd_workspace_size(dims)) return LOGO_ERR_WORKSPACE;
    const RowSet R{pos, cu_q, n_sel_total, dims.B, dims.T};
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    float* part = static_cast<float*>(workspace);
    if (a_lp && !pos && dims.D == 128)  // every row: the tcgen05 pipeline
        return launch_lp_tc_bwd(u_l, a_lp, du_g, dims, du_l, accumulate, da_lp, part, st);
    if (a_lp) {
        return dims.D == 128 ? launch_lp_bwd<128>(u_l, a_lp, du_g, R, dims.Hq, du_l, accumulate, da_lp, part, st)
                             : launch_lp_bwd<64>(u_l, a_lp, du_g, R, dims.Hq, du_l, accumulate, da_lp, part, st);
    }
    const int grid = so_bwd_blocks(dims);
    switch (so_vpt(dims)) {
        case 1: so_bwd_kernel<1><<<grid, 256, 0, st>>>(u_l, s_so, du_g, R, dims.Hq, dims.D, du_l, accumulate, part); break;
        case 2: so_bwd_kernel<2><<<grid, 256, 0, st>>>(u_l, s_so, du_g, R, dims.Hq, dims.D, du_l, accumulate, part); break;
        default: so_bwd_kernel<4><<<grid, 256, 0, st>>>(u_l, s_so, du_g, R, dims.Hq, dims.D, du_l, accumulate, part); break;
    }
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    const int hd = dims.Hq * dims.D;
    colsum_kernel<<<colsum_blocks(2 * hd), kColSumThreads, 0, st>>>(part, grid, 2 * hd, hd, ds_so, db_so);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
