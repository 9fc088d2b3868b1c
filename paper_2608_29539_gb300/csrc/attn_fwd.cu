// attn_fwd.cu -- forward of both attention branches on tcgen05 tensor cores.
//
//   logo_local_attn_fwd          O^L = SoftmaxAttn_W(Q^L, K^L, V^L)   (Eq. 6)
//   logo_global_sparse_attn_fwd  O^G_I = SoftmaxAttn_inf(Q^G_I, K^G, V^G) (Eq. 8)
//
// One persistent kernel template serves both.  A CTA (12 warps) loops over
// work items = (128-row query tile, query head):
//   warp 8      TMA producer: Q tile once per item, then K blocks (local: K
//               and V blocks) through a ring of shared-memory stages
//               (128-byte swizzle)
//   warp 11     global branch: V blocks through a ring of their own
//   warp 9      S issuer (one thread): S = Q K^T into one of two TMEM S buffers
//   warp 10     P.V issuer (one thread): O += P V into the TMEM O accumulator
//               with P read straight from TMEM.  Two issuing threads keep the
//               tensor pipe fed while either waits for its inputs: the issue
//               queue is short, so a single thread that stops to wait starves
//               the pipe (measured: 1728 vs 2427 TFLOP/s on the same MMA stream).
//   warps 0..3  softmax: one thread per query row (its TMEM lane).  Online
//               softmax in the log2 domain with conditional rescaling of O
//               (only when the running max grows by more than 2^8); P goes
//               back to TMEM as bf16 pairs, into one of two P buffers, so the
//               softmax of block n never waits for the P.V of block n-1
//               unless it has to rescale O.
//   warps 4..7  epilogue: O out of TMEM once an item's last P.V is done,
//               normalised and stored while the softmax warps start the next
//               item.
// The KV blocks of an item are only those some row can see; blocks where
// every row sees every key skip the per-element predicate (App. B's
// three-region traversal; for the local branch the window edge is a second
// masked region), and inside a masked block only the 32-key groups a row
// sees in part are tested key by key.  Global items come from a schedule
// ordered by cost (longest first) that a one-block kernel builds on the
// device, so nothing here needs the selected count on the host.
#include <cuda_bf16.h>

#include <cstdint>

#include "attn_common.cuh"
#include "host_common.h"
#include "sm100.cuh"

namespace logo {
namespace {

template <int D>
struct FwdCfg {
    static constexpr int kSub = D / 64;             // 64-column (128-byte) sub-tiles per row
    static constexpr int kTileBytes = kBM * D * 2;  // one Q / K / V tile
    // K/V ring of three stages.  The global branch runs K and V as two rings
    // with a producer each: a K stage is free once S of its block is done, a
    // V stage once P.V is, so K loads run further ahead (global fwd -7% at
    // 16K).  The local branch keeps one producer loading K and V of a block
    // together into one stage that P.V frees (its short items ran 6% slower
    // with the split).
    static constexpr int kStages = 3;
    static constexpr int kOffQ = 0;
    static constexpr int kOffK = kOffQ + kTileBytes;
    static constexpr int kOffV = kOffK + kStages * kTileBytes;
    static constexpr int kSmemBytes = kOffV + kStages * kTileBytes + 1024;  // + alignment slack
    static constexpr uint32_t kColO = 0;     // O accumulator (D columns, fp32)
    static constexpr uint32_t kColS0 = 128;  // S buffers (128 columns, fp32)
    static constexpr uint32_t kColS1 = 256;
    static constexpr uint32_t kColP0 = 384;  // P buffers (128 keys as bf16 pairs: 64 columns)
    static constexpr uint32_t kColP1 = 448;
    static constexpr uint32_t kTmemCols = 512;
    // 12 warps: softmax (0..3), epilogue (4..7), Q/K(/V) producer, S issuer,
    // P.V issuer, global branch: V producer (8..11).  Launched at 168 registers a thread (384 x 168 =
    // 64,512); the softmax warpgroup takes 224 (its row of S lives in
    // registers), the epilogue 168 (a row of O), the control warps 88:
    // 128 x (224 + 168 + 88) = 61,440.
    static constexpr int kThreads = 384;
    static constexpr uint32_t kRegsSoftmax = 224;
    static constexpr uint32_t kRegsEpilogue = 168;
    static constexpr uint32_t kRegsControl = 88;
};

struct FwdParams {
    CUtensorMap tm_q;  // local: Q [B,T,Hq,D]; global: packed Qc [1,cap+128,Hq,D]
    CUtensorMap tm_k;  // [B,T,Hkv,D]
    CUtensorMap tm_v;
    logo_bf16* o;      // local: [B,T,Hq,D]; global: packed [cap,Hq,D]
    float* lse;        // local: [B,Hq,T];   global: [Hq,cap]
    const int32_t* pos;            // global: packed positions
    const GlobalTile* tiles;       // global: schedule
    const int32_t* n_tiles;        // global: schedule length (device)
    int32_t* next_item;            // global: work counter, zeroed by the schedule kernel
    float* o_part;                 // global split entries: unnormalised O [slot * Hq + h][D][128]
    float* m_part;                 // ... their running max (log2 units) [slot * Hq + h][128]
    float* l_part;                 // ... and their row sums
    int B, T, Hq, Hkv, window, cap;
    int q_tiles;                   // local: query tiles per sequence
    float scale_log2;              // softmax scale * log2(e)
};

template <bool GLOBAL>
__device__ __forceinline__ FwdItem decode_item(const FwdParams& p, int k)
{
    FwdItem it;
    it.h = k % p.Hq;
    it.kvh = it.h / (p.Hq / p.Hkv);
    const int tile = k / p.Hq;
    if (!GLOBAL) {
        it.b = tile / p.q_tiles;
        const int qt = tile % p.q_tiles;
        it.row0 = qt * kBM;
        it.nrows = min(kBM, p.T - it.row0);
        it.pos_min = it.row0;
        it.pos_max = it.row0 + it.nrows - 1;
        it.blk_lo = max(0, it.pos_min - p.window + 1) / kBN;
        it.blk_hi = it.pos_max / kBN;
        it.slot = -1;
    } else {
        const GlobalTile g = p.tiles[tile];
        it.b = g.b;
        it.row0 = g.row0;
        it.nrows = g.nrows;
        it.pos_min = g.min_pos;
        it.pos_max = g.max_pos;
        it.blk_lo = g.blk_lo;
        it.blk_hi = g.blk_hi;
        it.slot = g.slot;
    }
    return it;
}

// Visibility inside one 128-key block: the row sees keys c with lo <= c <= hi;
// every other s[c] becomes -inf.  Called by all 32 lanes of a warp, whose rows
// are consecutive, so most 32-key groups are seen whole by every row of the
// warp or by none of them; one warp reduction classifies the groups.  Selects
// and moves cost two issue cycles per warp on this pipe, so only the groups
// in between get the per-key select, and only against the bound that cuts
// them; unseen groups get plain moves.
__device__ __forceinline__ void mask_row_block(float (&s)[kBN], int lo, int hi)
{
    uint32_t cls = 0;  // per group g: bit g seen whole, 4+g unseen, 8+g lo does not cut, 12+g hi does not cut
#pragma unroll
    for (int g = 0; g < kBN / 32; ++g) {
        const bool lo_cuts = lo > 32 * g, hi_cuts = hi < 32 * g + 31;
        cls |= (!lo_cuts && !hi_cuts) ? (1u << g) : 0u;
        cls |= (hi < 32 * g || lo > 32 * g + 31) ? (16u << g) : 0u;
        cls |= lo_cuts ? 0u : (256u << g);
        cls |= hi_cuts ? 0u : (4096u << g);
    }
    cls = __reduce_and_sync(0xffffffffu, cls);
#pragma unroll
    for (int g = 0; g < kBN / 32; ++g) {
        if (cls & (1u << g)) continue;
        if (cls & (16u << g)) {
            // (an opaque move: a constant assigned in this branch made the
            // compiler spill the row)
#pragma unroll
            for (int i = 0; i < 32; ++i) asm volatile("mov.b32 %0, 0xff800000;" : "=f"(s[32 * g + i]));
        } else if (cls & (256u << g)) {
#pragma unroll
            for (int i = 0; i < 32; ++i) s[32 * g + i] = 32 * g + i <= hi ? s[32 * g + i] : -INFINITY;
        } else if (cls & (4096u << g)) {
#pragma unroll
            for (int i = 0; i < 32; ++i) s[32 * g + i] = 32 * g + i >= lo ? s[32 * g + i] : -INFINITY;
        } else {
#pragma unroll
            for (int i = 0; i < 32; ++i)
                s[32 * g + i] = (32 * g + i >= lo && 32 * g + i <= hi) ? s[32 * g + i] : -INFINITY;
        }
    }
}

template <int D, bool GLOBAL>
__global__ void __launch_bounds__(384, 1) attn_fwd_kernel(const __grid_constant__ FwdParams p)
{
    using C = FwdCfg<D>;
    static_assert(128 * (C::kRegsSoftmax + C::kRegsEpilogue + C::kRegsControl) <= 384 * 168,
                  "register split exceeds the launch allocation");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    __shared__ __align__(8) uint64_t bar_q_full, bar_q_empty, bar_drain, bar_drain_pv;
    // bar_k_empty frees a K stage (global) or a K/V stage (local); bar_v_empty
    // a V stage (global only)
    __shared__ __align__(8) uint64_t bar_k_full[C::kStages], bar_k_empty[C::kStages];
    __shared__ __align__(8) uint64_t bar_v_full[C::kStages], bar_v_empty[C::kStages];
    __shared__ __align__(8) uint64_t bar_s_full[2], bar_s_empty[2], bar_p_full[2], bar_p_free[2];
    // softmax -> epilogue: 1/l of every row of an item (two slots), and O's
    // columns free again once the epilogue has copied them out
    __shared__ __align__(8) uint64_t bar_l_full[2], bar_l_empty[2], bar_o_free;
    __shared__ float sh_inv_l[2][kBM];
    __shared__ uint32_t tmem_base_sh;
    __shared__ volatile int abort_flag;
    // global branch: items are taken dynamically (longest first, whichever CTA
    // is free next); the producer passes each index to the other roles
    // through this 4-slot ring (-1 ends the work)
    __shared__ volatile int item_ring[4];
    __shared__ __align__(8) uint64_t bar_item_full[4], bar_item_empty[4];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t sQ = smem_u32(smem + C::kOffQ);
    const uint32_t sK = smem_u32(smem + C::kOffK);
    const uint32_t sV = smem_u32(smem + C::kOffV);

    if (threadIdx.x == 0) {
        abort_flag = 0;
        mbar_init(smem_u32(&bar_q_full), 1);
        mbar_init(smem_u32(&bar_q_empty), 1);
        mbar_init(smem_u32(&bar_drain), 1);
        mbar_init(smem_u32(&bar_drain_pv), 1);
        for (int s = 0; s < C::kStages; ++s) {
            mbar_init(smem_u32(&bar_k_full[s]), 1);
            mbar_init(smem_u32(&bar_k_empty[s]), 1);
            mbar_init(smem_u32(&bar_v_full[s]), 1);
            mbar_init(smem_u32(&bar_v_empty[s]), 1);
        }
        for (int s = 0; s < 4; ++s) {
            mbar_init(smem_u32(&bar_item_full[s]), 1);
            // the V producer, the two MMA threads, one lane per softmax / epilogue warp
            mbar_init(smem_u32(&bar_item_empty[s]), 11);
        }
        for (int s = 0; s < 2; ++s) {
            mbar_init(smem_u32(&bar_s_full[s]), 1);
            mbar_init(smem_u32(&bar_s_empty[s]), 128);
            mbar_init(smem_u32(&bar_p_full[s]), 128);
            mbar_init(smem_u32(&bar_p_free[s]), 1);
            mbar_init(smem_u32(&bar_l_full[s]), 128);
            mbar_init(smem_u32(&bar_l_empty[s]), 128);
        }
        mbar_init(smem_u32(&bar_o_free), 128);
        fence_mbar_init();
    }
    if (warp == 9) {
        tmem_alloc(smem_u32(&tmem_base_sh), C::kTmemCols);
        tmem_relinquish();
    }
    const int n_items = GLOBAL ? (*p.n_tiles) * p.Hq : p.B * p.q_tiles * p.Hq;
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_base_sh;

    // u-th work item of this CTA for a consumer role, or -1 when done.
    // whole_warp: called by all 32 lanes (the softmax warps), which then
    // arrive once per warp; otherwise by the single MMA-issuing thread.
    auto consume_item = [&](int u, bool* ok, bool whole_warp) -> int {
        if (!GLOBAL) {
            const int k = blockIdx.x + u * gridDim.x;
            return k < n_items ? k : -1;
        }
        const int slot = u & 3;
        if (!(*ok = mbar_wait(smem_u32(&bar_item_full[slot]), (u >> 2) & 1, &abort_flag))) return -1;
        const int k = item_ring[slot];
        if (whole_warp) {
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_u32(&bar_item_empty[slot]));
        } else {
            mbar_arrive(smem_u32(&bar_item_empty[slot]));
        }
        return k;
    };

    if (warp >= 8) {
        // ------------------------------------------------------------ control warps
        setmaxnreg_dec<C::kRegsControl>();
    if (warp == 8) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            tma_prefetch_desc(&p.tm_q);
            tma_prefetch_desc(&p.tm_k);
            tma_prefetch_desc(&p.tm_v);
            const uint64_t pol_q = policy_evict_first();
            const uint64_t pol_kv = policy_evict_last();
            int kv_it = 0, item_i = 0;
            int last_fill[C::kStages];
            for (int s = 0; s < C::kStages; ++s) last_fill[s] = -1;
            int q_fills = 0;
            bool ok = true;
            for (;; ++item_i) {
                int k;
                if (GLOBAL) {
                    const int slot = item_i & 3;
                    if (!(ok = mbar_wait(smem_u32(&bar_item_empty[slot]), ((item_i >> 2) & 1) ^ 1, &abort_flag))) break;
                    k = atomicAdd(p.next_item, 1);
                    if (k >= n_items) k = -1;
                    item_ring[slot] = k;
                    mbar_arrive(smem_u32(&bar_item_full[slot]));
                } else {
                    k = blockIdx.x + item_i * gridDim.x;
                    if (k >= n_items) k = -1;
                }
                if (k < 0) break;
                const FwdItem it = decode_item<GLOBAL>(p, k);
                if (!(ok = mbar_wait(smem_u32(&bar_q_empty), (item_i & 1) ^ 1, &abort_flag))) break;
                const uint32_t qb = smem_u32(&bar_q_full);
                mbar_arrive_expect_tx(qb, C::kTileBytes);
                for (int s = 0; s < C::kSub; ++s)
                    tma_load_4d(sQ + s * 16384, &p.tm_q, qb, 64 * s, it.h, it.row0, GLOBAL ? 0 : it.b, pol_q);
                ++q_fills;
                for (int n = it.blk_lo; n <= it.blk_hi; ++n, ++kv_it) {
                    const int st = kv_it % C::kStages, f = kv_it / C::kStages;
                    if (!(ok = mbar_wait(smem_u32(&bar_k_empty[st]), (f & 1) ^ 1, &abort_flag))) break;
                    const uint32_t kb = smem_u32(&bar_k_full[st]);
                    mbar_arrive_expect_tx(kb, C::kTileBytes);
                    for (int s = 0; s < C::kSub; ++s)
                        tma_load_4d(sK + st * C::kTileBytes + s * 16384, &p.tm_k, kb, 64 * s, it.kvh, n * kBN, it.b,
                                    pol_kv);
                    if (!GLOBAL) {  // V of the same block into the same stage
                        const uint32_t vb = smem_u32(&bar_v_full[st]);
                        mbar_arrive_expect_tx(vb, C::kTileBytes);
                        for (int s = 0; s < C::kSub; ++s)
                            tma_load_4d(sV + st * C::kTileBytes + s * 16384, &p.tm_v, vb, 64 * s, it.kvh, n * kBN,
                                        it.b, pol_kv);
                    }
                    last_fill[st] = f;
                }
                if (!ok) break;
            }
            if (!ok) {  // let copies already issued land before the CTA exits
                if (q_fills > 0) mbar_wait_drain(smem_u32(&bar_q_full), (q_fills - 1) & 1);
                for (int s = 0; s < C::kStages; ++s)
                    if (last_fill[s] >= 0) {
                        mbar_wait_drain(smem_u32(&bar_k_full[s]), last_fill[s] & 1);
                        if (!GLOBAL) mbar_wait_drain(smem_u32(&bar_v_full[s]), last_fill[s] & 1);
                    }
            }
        }
    } else if (warp == 9) {
        // ------------------------------------------------------------ S issuer
        // S = Q K^T of every block; the P.V products come from warp 6, so that
        // neither stream's waits leave the tensor pipe without queued work
        // (the issue queue is short: an issuing thread runs only a few
        // instructions ahead of execution)
        if (lane == 0) {
            constexpr uint32_t idS = idesc_bf16_f32(kBM, kBN, false, false);
            int kv_it = 0, s_it = 0, item_i = 0;
            bool ok = true;
            for (;; ++item_i) {
                const int k = consume_item(item_i, &ok, false);
                if (k < 0) break;
                const FwdItem it = decode_item<GLOBAL>(p, k);
                const int nblk = it.blk_hi - it.blk_lo + 1;
                if (!(ok = mbar_wait(smem_u32(&bar_q_full), item_i & 1, &abort_flag))) break;
                for (int j = 0; j < nblk && ok; ++j) {
                    const int itg = s_it + j;
                    const int st = (kv_it + j) % C::kStages, f = (kv_it + j) / C::kStages;
                    const int buf = itg & 1, use = itg >> 1;
                    if (!(ok = mbar_wait(smem_u32(&bar_k_full[st]), f & 1, &abort_flag))) break;
                    if (!(ok = mbar_wait(smem_u32(&bar_s_empty[buf]), (use & 1) ^ 1, &abort_flag))) break;
                    tc_fence_after();
                    const uint32_t kbase = sK + st * C::kTileBytes;
                    const uint32_t dcol = tmem + (buf ? C::kColS1 : C::kColS0);
#pragma unroll
                    for (int ks = 0; ks < D / 16; ++ks) {
                        const uint32_t off = (ks >> 2) * 16384 + (ks & 3) * 32;
                        umma_bf16_ss(dcol, sdesc_sw128(sQ + off, 16, 1024), sdesc_sw128(kbase + off, 16, 1024), idS,
                                     ks > 0 ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_s_full[buf]));
                    if (GLOBAL) umma_commit(smem_u32(&bar_k_empty[st]));  // K of this block is read
                }
                if (!ok) break;
                umma_commit(smem_u32(&bar_q_empty));
                kv_it += nblk;
                s_it += nblk;
            }
            if (!ok) {  // wait for MMAs in flight before TMEM is released
                umma_commit(smem_u32(&bar_drain));
                mbar_wait_drain(smem_u32(&bar_drain), 0);
            }
        }
    } else if (warp == 10) {
        // ------------------------------------------------------------ P.V issuer
        if (lane == 0) {
            constexpr uint32_t idPV = idesc_bf16_f32(kBM, D, false, true);
            int kv_it = 0, s_it = 0, item_i = 0;
            bool ok = true;
            for (;; ++item_i) {
                const int k = consume_item(item_i, &ok, false);
                if (k < 0) break;
                const FwdItem it = decode_item<GLOBAL>(p, k);
                const int nblk = it.blk_hi - it.blk_lo + 1;
                for (int j = 0; j < nblk && ok; ++j) {
                    const int itg = s_it + j;
                    const int st = (kv_it + j) % C::kStages, f = (kv_it + j) / C::kStages;
                    if (!(ok = mbar_wait(smem_u32(&bar_p_full[itg & 1]), (itg >> 1) & 1, &abort_flag))) break;
                    if (!(ok = mbar_wait(smem_u32(&bar_v_full[st]), f & 1, &abort_flag))) break;
                    // the item's first P.V overwrites O: the epilogue warps have
                    // copied the previous item's O out of TMEM
                    if (j == 0 && !(ok = mbar_wait(smem_u32(&bar_o_free), (item_i & 1) ^ 1, &abort_flag))) break;
                    tc_fence_after();
                    const uint32_t vbase = sV + st * C::kTileBytes;
                    const uint32_t pcol = tmem + ((itg & 1) ? C::kColP1 : C::kColP0);
#pragma unroll
                    for (int ks = 0; ks < kBN / 16; ++ks) {
                        const uint64_t bdesc = sdesc_sw128(vbase + ks * 2048, 16384, 1024);
                        umma_bf16_ts(tmem + C::kColO, pcol + ks * 8, bdesc, idPV, (j > 0 || ks > 0) ? 1u : 0u);
                    }
                    umma_commit(smem_u32(&bar_p_free[itg & 1]));
                    // V of this block is read (local: K and V, whose S was done before P)
                    umma_commit(smem_u32(GLOBAL ? &bar_v_empty[st] : &bar_k_empty[st]));
                }
                if (!ok) break;
                kv_it += nblk;
                s_it += nblk;
            }
            if (!ok) {
                umma_commit(smem_u32(&bar_drain_pv));
                mbar_wait_drain(smem_u32(&bar_drain_pv), 0);
            }
        }
    } else if (GLOBAL && warp == 11) {
        // ------------------------------------------------------------ V producer
        // global branch: V blocks through their own ring (a stage is freed by
        // the P.V that read it), so a V load never holds up the next K load
        if (lane == 0) {
            const uint64_t pol_kv = policy_evict_last();
            int kv_it = 0;
            int last_fill[C::kStages];
            for (int s = 0; s < C::kStages; ++s) last_fill[s] = -1;
            bool ok = true;
            for (int item_i = 0;; ++item_i) {
                const int k = consume_item(item_i, &ok, false);
                if (k < 0) break;
                const FwdItem it = decode_item<GLOBAL>(p, k);
                for (int n = it.blk_lo; n <= it.blk_hi; ++n, ++kv_it) {
                    const int st = kv_it % C::kStages, f = kv_it / C::kStages;
                    if (!(ok = mbar_wait(smem_u32(&bar_v_empty[st]), (f & 1) ^ 1, &abort_flag))) break;
                    const uint32_t vb = smem_u32(&bar_v_full[st]);
                    mbar_arrive_expect_tx(vb, C::kTileBytes);
                    for (int s = 0; s < C::kSub; ++s)
                        tma_load_4d(sV + st * C::kTileBytes + s * 16384, &p.tm_v, vb, 64 * s, it.kvh, n * kBN, it.b,
                                    pol_kv);
                    last_fill[st] = f;
                }
                if (!ok) break;
            }
            if (!ok) {  // let copies already issued land before the CTA exits
                for (int s = 0; s < C::kStages; ++s)
                    if (last_fill[s] >= 0) mbar_wait_drain(smem_u32(&bar_v_full[s]), last_fill[s] & 1);
            }
        }
    }
    } else if (warp < 4) {
        // ------------------------------------------------------------ softmax
        setmaxnreg_inc<C::kRegsSoftmax>();
        const int quad = warp & 3;  // TMEM lane quadrant this warp may access
        const int r = quad * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        const int window = GLOBAL ? kNoWindow : p.window;
        int itg = 0;
        bool ok = true;
        for (int item_i = 0;; ++item_i) {
            const int k = consume_item(item_i, &ok, true);
            if (k < 0) break;
            const FwdItem it = decode_item<GLOBAL>(p, k);
            const bool row_valid = r < it.nrows;
            int mypos;
            if (GLOBAL) mypos = row_valid ? p.pos[it.row0 + r] : it.pos_max;
            else mypos = row_valid ? it.row0 + r : it.pos_max;
            float m_ref = -INFINITY;  // running max, log2 domain
            float l = 0.f;
            // The S-ready and P-buffer-free barriers are nearly always complete
            // by the time they are needed; each is tested (non-blocking) well
            // before that point, so the test's latency overlaps other work, and
            // only a warp that found one incomplete waits on it.
            bool s_ready = false;  // S of this block seen complete while the previous block ended
            for (int n = it.blk_lo; n <= it.blk_hi; ++n, ++itg) {
                const int buf = itg & 1, use = itg >> 1;
                if (!s_ready) {
                    ok = mbar_wait(smem_u32(&bar_s_full[buf]), use & 1, &abort_flag);
                    __syncwarp();
                    if (!ok) break;
                }
                tc_fence_after();
                float s[kBN];
                const uint32_t scol = tmem + lane_off + (buf ? C::kColS1 : C::kColS0);
                {
                    uint32_t v[kBN / 32][32];
#pragma unroll
                    for (int c = 0; c < kBN / 32; ++c) tmem_ld32(scol + c * 32, v[c]);
                    tmem_wait_ld();  // one wait for all four loads
#pragma unroll
                    for (int c = 0; c < kBN / 32; ++c)
#pragma unroll
                        for (int i = 0; i < 32; ++i) s[c * 32 + i] = __uint_as_float(v[c][i]);
                }
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_s_empty[buf]));
                // P buffer itg%2 is free once the P.V two blocks back is done
                const bool p_free_seen = mbar_test(smem_u32(&bar_p_free[itg & 1]), ((itg >> 1) & 1) ^ 1);
                if (block_needs_mask(n, it.pos_min, it.pos_max, window))
                    mask_row_block(s, mypos - window + 1 - n * kBN, mypos - n * kBN);
                // 4 independent 3-input max chains and 4 packed-pair sums keep
                // dependency chains short; exp arguments are formed two at a
                // time with f32x2 FMAs
                float mx4[4] = {s[0], s[1], s[2], s[3]};
#pragma unroll
                for (int c = 4; c < kBN; c += 8) {
                    mx4[0] = max3f(mx4[0], s[c], s[c + 1]);
                    mx4[1] = max3f(mx4[1], s[c + 2], s[c + 3]);
                    if (c + 4 < kBN) {
                        mx4[2] = max3f(mx4[2], s[c + 4], s[c + 5]);
                        mx4[3] = max3f(mx4[3], s[c + 6], s[c + 7]);
                    }
                }
                const float mx = max3f(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3]));
                const float m_new = fmaxf(m_ref, mx * p.scale_log2);
                float alpha = 1.f;
                bool rescale = false;
                if (m_new > m_ref + 8.0f) {  // also taken when m_ref is still -inf
                    alpha = ex2_approx(m_ref - m_new);
                    m_ref = m_new;
                    rescale = true;
                }
                const float m_use = (m_ref == -INFINITY) ? 0.f : m_ref;
                const uint64_t scale2 = f2_pack(p.scale_log2, p.scale_log2);
                const uint64_t negm2 = f2_pack(-m_use, -m_use);
                uint64_t acc2[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
                for (int c = 0; c < kBN; c += 2) {
                    float x0, x1;
                    f2_unpack(f2_fma(f2_pack(s[c], s[c + 1]), scale2, negm2), x0, x1);
                    s[c] = ex2_approx(x0);
                    s[c + 1] = ex2_approx(x1);
                    acc2[(c >> 1) & 3] = f2_add(acc2[(c >> 1) & 3], f2_pack(s[c], s[c + 1]));
                }
                float rs;
                {
                    float a0, a1, b0, b1, c0, c1, d0, d1;
                    f2_unpack(acc2[0], a0, a1);
                    f2_unpack(acc2[1], b0, b1);
                    f2_unpack(acc2[2], c0, c1);
                    f2_unpack(acc2[3], d0, d1);
                    rs = ((a0 + a1) + (b0 + b1)) + ((c0 + c1) + (d0 + d1));
                }
                l = l * alpha + rs;
                // O may only be rescaled once the P.V of the previous block is done
                const bool warp_rescale = __any_sync(0xffffffffu, rescale && n > it.blk_lo);
                if (warp_rescale) {
                    // P.V of block itg-1 done: the completion on its P buffer
                    // (unambiguous: the one before it was awaited a block ago)
                    ok = mbar_wait(smem_u32(&bar_p_free[(itg - 1) & 1]), ((itg - 1) >> 1) & 1, &abort_flag);
                    __syncwarp();
                    if (!ok) break;
                    tc_fence_after();
                    // tcgen05.ld/st are warp-collective: rows that keep their max
                    // multiply by alpha = 1
                    const uint32_t ocol = tmem + lane_off + C::kColO;
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t v[32];
                        tmem_ld32(ocol + c * 32, v);
                        tmem_wait_ld();
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = __float_as_uint(__uint_as_float(v[i]) * alpha);
                        tmem_st32(ocol + c * 32, v);
                    }
                }
                if (!__all_sync(0xffffffffu, p_free_seen)) {
                    ok = mbar_wait(smem_u32(&bar_p_free[itg & 1]), ((itg >> 1) & 1) ^ 1, &abort_flag);
                    __syncwarp();
                    if (!ok) break;
                }
                tc_fence_after();
                const uint32_t pcol = tmem + lane_off + ((itg & 1) ? C::kColP1 : C::kColP0);
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    uint32_t pk[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) pk[i] = cvt_bf16x2(s[64 * h + 2 * i], s[64 * h + 2 * i + 1]);
                    tmem_st32(pcol + 32 * h, pk);
                }
                const bool s_seen = n < it.blk_hi && mbar_test(smem_u32(&bar_s_full[(itg + 1) & 1]), ((itg + 1) >> 1) & 1);
                tmem_wait_st();
                tc_fence_before();
                mbar_arrive(smem_u32(&bar_p_full[itg & 1]));
                s_ready = __all_sync(0xffffffffu, s_seen);
            }
            if (!ok) break;
            // ---- end of the item: lse = (m + log2 l) ln 2, and 1/l to the
            //      epilogue warps, which normalise O while this warp moves on
            if (row_valid) {
                const float lse = (m_ref + log2f(l)) * kLn2;
                if (GLOBAL && it.slot < 0) p.lse[static_cast<int64_t>(it.h) * p.cap + it.row0 + r] = lse;
                else if (!GLOBAL) p.lse[(static_cast<int64_t>(it.b) * p.Hq + it.h) * p.T + it.row0 + r] = lse;
            }
            const int ls = item_i & 1;
            ok = mbar_wait(smem_u32(&bar_l_empty[ls]), ((item_i >> 1) & 1) ^ 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            // a share of a split KV range hands over its row sum (the merge
            // normalises); everything else 1/l
            sh_inv_l[ls][r] = (GLOBAL && it.slot >= 0) ? l : 1.0f / l;
            if (GLOBAL && it.slot >= 0 && row_valid)
                p.m_part[(static_cast<int64_t>(it.slot) * p.Hq + it.h) * kBM + r] = m_ref;
            mbar_arrive(smem_u32(&bar_l_full[ls]));
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // warps 4..7: once an item's last P.V is done, copy O out of TMEM (then
        // the next item's first P.V may overwrite it), and write O / l (or, for
        // one share of a split KV range, the unnormalised O and the row sum)
        setmaxnreg_dec<C::kRegsEpilogue>();
        const int quad = warp & 3;
        const int r = quad * 32 + lane;
        const uint32_t lane_off = static_cast<uint32_t>(quad * 32) << 16;
        int itg = 0;
        bool ok = true;
        for (int item_i = 0;; ++item_i) {
            const int k = consume_item(item_i, &ok, true);
            if (k < 0) break;
            const FwdItem it = decode_item<GLOBAL>(p, k);
            const bool row_valid = r < it.nrows;
            itg += it.blk_hi - it.blk_lo + 1;
            const int ls = item_i & 1;
            ok = mbar_wait(smem_u32(&bar_l_full[ls]), (item_i >> 1) & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            const float lv = sh_inv_l[ls][r];
            mbar_arrive(smem_u32(&bar_l_empty[ls]));
            // the item's last P.V (block itg - 1) is done
            ok = mbar_wait(smem_u32(&bar_p_free[(itg - 1) & 1]), ((itg - 1) >> 1) & 1, &abort_flag);
            __syncwarp();
            if (!ok) break;
            tc_fence_after();
            uint32_t ov[D / 32][32];
            const uint32_t ocol = tmem + lane_off + C::kColO;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) tmem_ld32(ocol + c * 32, ov[c]);
            tmem_wait_ld();
            tc_fence_before();
            mbar_arrive(smem_u32(&bar_o_free));
            if (GLOBAL && it.slot >= 0) {
                // one share of a split KV range: unnormalised O, stored transposed
                // ([d][row]) so that the warp's 32 rows of a column are one line
                const int64_t unit = static_cast<int64_t>(it.slot) * p.Hq + it.h;
                float* pcol = p.o_part + unit * kBM * D + r;
#pragma unroll
                for (int c = 0; c < D / 32; ++c)
#pragma unroll
                    for (int i = 0; i < 32; ++i) pcol[(c * 32 + i) * kBM] = __uint_as_float(ov[c][i]);
                if (row_valid) p.l_part[unit * kBM + r] = lv;
                continue;
            }
            if (!row_valid) continue;
            const float inv_l = lv;
            logo_bf16* orow;
            if (GLOBAL) orow = p.o + (static_cast<int64_t>(it.row0 + r) * p.Hq + it.h) * D;
            else orow = p.o + ((static_cast<int64_t>(it.b) * p.T + it.row0 + r) * p.Hq + it.h) * D;
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
#pragma unroll
                for (int q4 = 0; q4 < 4; ++q4) {
                    const uint32_t* v = ov[c] + 8 * q4;
                    uint4 w;
                    w.x = pack_bf16x2(__uint_as_float(v[0]) * inv_l, __uint_as_float(v[1]) * inv_l);
                    w.y = pack_bf16x2(__uint_as_float(v[2]) * inv_l, __uint_as_float(v[3]) * inv_l);
                    w.z = pack_bf16x2(__uint_as_float(v[4]) * inv_l, __uint_as_float(v[5]) * inv_l);
                    w.w = pack_bf16x2(__uint_as_float(v[6]) * inv_l, __uint_as_float(v[7]) * inv_l);
                    *reinterpret_cast<uint4*>(orow + c * 32 + q4 * 8) = w;
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 9) {
        tc_fence_after();
        tmem_dealloc(tmem, C::kTmemCols);
    }
}

// ---------------------------------------------------------------- global prep
// Split-K of the global forward.  When the selected rows make too few work
// items to fill the GPU (query tiles x heads < 2 x SMs: small sequences, high
// sparsity), long tiles are cut into shares of their KV range, each share a
// work item of its own that leaves its unnormalised O, row max and row sum in
// a slot; merge_splits_kernel then combines the shares of each row exactly
// (rescaling each share by 2^(m_s - M) to the common max M).  At most
// kMaxPartialUnits (slot, head) pairs of partial results exist.
constexpr int kMaxPartialUnits = 1024;
constexpr int kMinSplitBlocks = 8;
constexpr int kMaxShares = 64;  // shares of one tile
// Splitting pays only when it shortens the longest item by more than the merge
// and the extra items cost (measured: about a dozen blocks' time); below this
// many blocks of gain the tiles stay whole.
constexpr int kSplitMinGainBlocks = 24;

// One block: split every sequence's packed rows into tiles of 128, split long
// tiles' KV ranges if the tiles are too few, and order the entries by their
// KV-block count, longest first.
__device__ __forceinline__ int sched_block_scan(int v, int* total, int* sh)
{
    // exclusive scan over the 1024 threads, in thread order
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int x = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_up_sync(0xffffffffu, x, o);
        if (lane >= o) x += y;
    }
    if (lane == 31) sh[warp] = x;
    __syncthreads();
    if (warp == 0) {
        const int w0 = sh[lane];
        int w = w0;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int y = __shfl_up_sync(0xffffffffu, w, o);
            if (lane >= o) w += y;
        }
        sh[lane] = w - w0;
        if (lane == 31) sh[32] = w;
    }
    __syncthreads();
    const int r = sh[warp] + x - v;
    *total = sh[32];
    __syncthreads();
    return r;
}

__global__ void __launch_bounds__(1024) global_schedule_kernel(const int32_t* __restrict__ pos,
                                                               const int32_t* __restrict__ cu_q, int B, int Hq,
                                                               int n_sm, int32_t* __restrict__ tile_off,
                                                               GlobalTile* __restrict__ unsorted,
                                                               GlobalTile* __restrict__ sorted,
                                                               int32_t* __restrict__ n_tiles,
                                                               int32_t* __restrict__ next_item,
                                                               SplitTile* __restrict__ splits,
                                                               int32_t* __restrict__ n_splits)
{
    __shared__ int sh_nt, sh_chunk, sh_worth;
    __shared__ int sh_scan[33];
    __shared__ unsigned long long sh_total;
    __shared__ int sh_longest;
    if (threadIdx.x == 0) {
        int acc = 0;
        for (int b = 0; b < B; ++b) {
            tile_off[b] = acc;
            acc += (cu_q[b + 1] - cu_q[b] + kBM - 1) / kBM;
        }
        tile_off[B] = acc;
        sh_nt = acc;
        sh_total = 0;
        sh_longest = 0;
        *next_item = 0;
    }
    __syncthreads();
    const int nt = sh_nt;
    // few tiles to fill the GPU with: split the long ones (then nt < 2 x SMs <= 1024)
    const bool split = static_cast<int64_t>(nt) * Hq < 2ll * n_sm && Hq <= kMaxPartialUnits && nt <= 1024;
    auto make_tile = [&](int t) {
        int lo = 0, hi = B - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (tile_off[mid] <= t) lo = mid;
            else hi = mid - 1;
        }
        const int b = lo, i = t - tile_off[b];
        GlobalTile g;
        g.row0 = cu_q[b] + i * kBM;
        g.nrows = min(kBM, cu_q[b + 1] - g.row0);
        g.b = b;
        g.min_pos = pos[g.row0];
        g.max_pos = pos[g.row0 + g.nrows - 1];
        g.blk_lo = 0;
        g.blk_hi = g.max_pos / kBN;
        g.slot = -1;
        g.cost = g.blk_hi + 1;
        g.pad0 = g.pad1 = g.pad2 = 0;
        return g;
    };
    int ne = nt;
    if (!split) {
        for (int t = threadIdx.x; t < nt; t += blockDim.x) unsorted[t] = make_tile(t);
        if (threadIdx.x == 0) *n_splits = 0;
    } else {
        // thread t < nt holds tile t
        GlobalTile g{};
        if (threadIdx.x < nt) {
            g = make_tile(threadIdx.x);
            atomicAdd(&sh_total, static_cast<unsigned long long>(g.cost));
            atomicMax(&sh_longest, g.cost);
        }
        __syncthreads();
        if (threadIdx.x == 0) {
            // cut only what is longer than an even share of the work per SM (the
            // longest item bounds the launch; every extra item costs a pipeline
            // restart and a partial write), in shares of at least kMinSplitBlocks
            // blocks and at most kMaxShares per tile
            const long long even = (static_cast<long long>(sh_total) * Hq + n_sm - 1) / n_sm;
            int chunk = static_cast<int>(even > kMinSplitBlocks ? even : kMinSplitBlocks);
            chunk = max(chunk, (sh_longest + kMaxShares - 1) / kMaxShares);
            sh_chunk = chunk;
            sh_worth = sh_longest - chunk >= kSplitMinGainBlocks;
        }
        __syncthreads();
    }
    if (split && !sh_worth) {  // too little to gain: the whole tiles after all
        for (int t = threadIdx.x; t < nt; t += blockDim.x) unsorted[t] = make_tile(t);
        if (threadIdx.x == 0) *n_splits = 0;
    } else if (split) {
        GlobalTile g{};
        if (threadIdx.x < nt) g = make_tile(threadIdx.x);
        // grow the shares until the split tiles fit in the partial-result slots
        const int max_slots = kMaxPartialUnits / Hq;
        int sp = 1, slots = 0;
        for (;;) {
            const int chunk = sh_chunk;
            sp = threadIdx.x < nt ? (g.cost + chunk - 1) / chunk : 0;
            sched_block_scan(sp > 1 ? sp : 0, &slots, sh_scan);
            if (slots <= max_slots) break;
            if (threadIdx.x == 0) sh_chunk = chunk * 2;
            __syncthreads();
        }
        int n_entries, n_split_tiles;
        const int e0 = sched_block_scan(threadIdx.x < nt ? sp : 0, &n_entries, sh_scan);
        const int s0 = sched_block_scan(sp > 1 ? sp : 0, &slots, sh_scan);
        const int t0 = sched_block_scan(sp > 1 ? 1 : 0, &n_split_tiles, sh_scan);
        if (threadIdx.x < nt) {
            if (sp == 1) {
                unsorted[e0] = g;
            } else {
                splits[t0] = SplitTile{g.row0, g.nrows, s0, sp};
                for (int s = 0; s < sp; ++s) {
                    GlobalTile e = g;
                    e.blk_lo = static_cast<int>(static_cast<int64_t>(g.cost) * s / sp);
                    e.blk_hi = static_cast<int>(static_cast<int64_t>(g.cost) * (s + 1) / sp) - 1;
                    e.slot = s0 + s;
                    e.cost = e.blk_hi - e.blk_lo + 1;
                    unsorted[e0 + s] = e;
                }
            }
        }
        if (threadIdx.x == 0) *n_splits = n_split_tiles;
        ne = n_entries;
    }
    if (threadIdx.x == 0) *n_tiles = ne;
    __syncthreads();  // entries written
    for (int t = threadIdx.x; t < ne; t += blockDim.x) {
        const int c = unsorted[t].cost;
        int rank = 0;
        for (int u = 0; u < ne; ++u) {
            const int cu = unsorted[u].cost;
            rank += (cu > c) || (cu == c && u < t);
        }
        sorted[rank] = unsorted[t];
    }
}

// Combine the shares of every split tile: per (row, head), M = max_s m_s,
// L = sum_s 2^(m_s - M) l_s, O = sum_s 2^(m_s - M) O_s / L, lse = (M + log2 L)
// ln 2.  A share whose keys the row cannot see has m_s = -inf and weighs 0.
// Work unit = (split tile, head, group of 8 columns); a block of 128 threads
// (thread = row) takes units in a grid stride, so every unit's 8 x shares
// loads per row are spread over the whole GPU; the transposed partials make
// each of a warp's loads one 128-byte line.
template <int D>
__global__ void __launch_bounds__(128) merge_splits_kernel(const SplitTile* __restrict__ splits,
                                                           const int32_t* __restrict__ n_splits, int Hq, int cap,
                                                           const float* __restrict__ o_part,
                                                           const float* __restrict__ m_part,
                                                           const float* __restrict__ l_part,
                                                           logo_bf16* __restrict__ o, float* __restrict__ lse)
{
    constexpr int kGroups = D / 8;
    const int n_units = *n_splits * Hq * kGroups;
    const int r = threadIdx.x;
    for (int un = blockIdx.x; un < n_units; un += gridDim.x) {
        const int g = un % kGroups, pr = un / kGroups;
        const SplitTile st = splits[pr / Hq];
        const int h = pr % Hq;
        if (r >= st.nrows) continue;
        const int64_t unit0 = static_cast<int64_t>(st.slot0) * Hq + h;  // share s: unit0 + s * Hq
        float M = -INFINITY;
        for (int s = 0; s < st.nsplit; ++s) M = fmaxf(M, m_part[(unit0 + static_cast<int64_t>(s) * Hq) * kBM + r]);
        float L = 0.f;
        float acc[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = 0.f;
        for (int s = 0; s < st.nsplit; ++s) {
            const int64_t unit = unit0 + static_cast<int64_t>(s) * Hq;
            const float m = m_part[unit * kBM + r];
            const float w = m == -INFINITY ? 0.f : ex2_approx(m - M);
            L += w * l_part[unit * kBM + r];
            const float* src = o_part + unit * kBM * D + (g * 8) * kBM + r;
            float v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = src[e * kBM];
#pragma unroll
            for (int e = 0; e < 8; ++e) acc[e] += w * v[e];
        }
        const float inv = 1.0f / L;
        uint4 w4;
        w4.x = pack_bf16x2(acc[0] * inv, acc[1] * inv);
        w4.y = pack_bf16x2(acc[2] * inv, acc[3] * inv);
        w4.z = pack_bf16x2(acc[4] * inv, acc[5] * inv);
        w4.w = pack_bf16x2(acc[6] * inv, acc[7] * inv);
        *reinterpret_cast<uint4*>(o + (static_cast<int64_t>(st.row0 + r) * Hq + h) * D + g * 8) = w4;
        if (g == 0) lse[static_cast<int64_t>(h) * cap + st.row0 + r] = (M + log2f(L)) * kLn2;
    }
}

struct GlobalFwdWs {
    logo_bf16* qc;
    GlobalTile* unsorted;
    GlobalTile* sorted;
    int32_t* tile_off;
    int32_t* n_tiles;
    int32_t* next_item;
    int32_t* n_splits;
    SplitTile* splits;
    float* o_part;
    float* m_part;
    float* l_part;
};

size_t global_fwd_ws_layout(const logo_dims& d, char* base, GlobalFwdWs* ws)
{
    const size_t cap = static_cast<size_t>(d.B) * d.T;
    const size_t max_tiles = cap / kBM + d.B + 1;
    const size_t max_entries = max_tiles + kMaxPartialUnits;  // each split adds at most one entry per slot
    size_t off = 0;
    const size_t o_qc = off;
    off = round_up(off + (cap + kBM) * d.Hq * d.D * 2, 256);
    const size_t o_un = off;
    off = round_up(off + max_entries * sizeof(GlobalTile), 256);
    const size_t o_so = off;
    off = round_up(off + max_entries * sizeof(GlobalTile), 256);
    const size_t o_to = off;
    off = round_up(off + (d.B + 1) * sizeof(int32_t), 256);
    const size_t o_nt = off;
    off = round_up(off + 4 * sizeof(int32_t), 256);
    const size_t o_sp = off;
    off = round_up(off + max_tiles * sizeof(SplitTile), 256);
    const size_t o_op = off;
    off = round_up(off + static_cast<size_t>(kMaxPartialUnits) * kBM * d.D * sizeof(float), 256);
    const size_t o_mp = off;
    off = round_up(off + static_cast<size_t>(kMaxPartialUnits) * kBM * sizeof(float), 256);
    const size_t o_lp = off;
    off = round_up(off + static_cast<size_t>(kMaxPartialUnits) * kBM * sizeof(float), 256);
    if (ws) {
        ws->qc = reinterpret_cast<logo_bf16*>(base + o_qc);
        ws->unsorted = reinterpret_cast<GlobalTile*>(base + o_un);
        ws->sorted = reinterpret_cast<GlobalTile*>(base + o_so);
        ws->tile_off = reinterpret_cast<int32_t*>(base + o_to);
        ws->n_tiles = reinterpret_cast<int32_t*>(base + o_nt);
        ws->next_item = ws->n_tiles + 1;
        ws->n_splits = ws->n_tiles + 2;
        ws->splits = reinterpret_cast<SplitTile*>(base + o_sp);
        ws->o_part = reinterpret_cast<float*>(base + o_op);
        ws->m_part = reinterpret_cast<float*>(base + o_mp);
        ws->l_part = reinterpret_cast<float*>(base + o_lp);
    }
    return off;
}

template <int D, bool GLOBAL>
int launch_fwd(const FwdParams& prm, int n_items_upper, cudaStream_t st)
{
    using C = FwdCfg<D>;
    static bool attr_done = false;  // benign race: setting the attribute twice is harmless
    if (!attr_done) {
        if (set_smem_limit(attn_fwd_kernel<D, GLOBAL>, C::kSmemBytes) != cudaSuccess) return LOGO_ERR_CUDA;
        attr_done = true;
    }
    const int grid = max(1, min(n_items_upper, device_sm_count()));
    attn_fwd_kernel<D, GLOBAL><<<grid, C::kThreads, C::kSmemBytes, st>>>(prm);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}

int check_attn_ptrs(const void* q, const void* k, const void* v)
{
    if (!q || !k || !v) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k) || !aligned16(v)) return LOGO_ERR_UNSUPPORTED;
    return LOGO_OK;
}

}  // namespace

int attn_fwd_tu_status(int clear) { return read_tu_status(clear); }

}  // namespace logo

using namespace logo;

extern "C" int logo_local_attn_fwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, logo_bf16* o,
                                   float* lse, logo_dims dims, int window, float scale, void* stream)
{
    int rc = check_dims(dims);
    if (rc != LOGO_OK) return rc;
    if ((rc = check_attn_ptrs(q, k, v)) != LOGO_OK) return rc;
    if (!o || !lse || window < 1) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(o)) return LOGO_ERR_UNSUPPORTED;
    if (!(scale >= 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (scale == 0.0f) scale = 1.0f / sqrtf(static_cast<float>(dims.D));
    FwdParams prm{};
    const int w = window > dims.T ? dims.T : window;
    if (!encode_bf16_4d(&prm.tm_q, q, dims.D, dims.Hq, dims.T, dims.B, 64, kBM) ||
        !encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN))
        return LOGO_ERR_CUDA;
    prm.o = o;
    prm.lse = lse;
    prm.B = dims.B;
    prm.T = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = w;
    prm.cap = dims.B * dims.T;
    prm.q_tiles = (dims.T + kBM - 1) / kBM;
    prm.scale_log2 = scale * kLog2e;
    const int n_items = dims.B * prm.q_tiles * dims.Hq;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    return dims.D == 128 ? launch_fwd<128, false>(prm, n_items, st) : launch_fwd<64, false>(prm, n_items, st);
}

extern "C" size_t logo_global_attn_fwd_workspace_size(logo_dims dims)
{
    if (check_dims(dims) != LOGO_OK) return 0;
    return global_fwd_ws_layout(dims, nullptr, nullptr);
}

extern "C" int logo_global_sparse_attn_fwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v,
                                           const int32_t* pos, const int32_t* cu_q, const int32_t* n_sel_total,
                                           logo_bf16* o_c, float* lse_c, logo_dims dims, float scale,
                                           void* workspace, size_t workspace_bytes, void* stream)
{
    int rc = check_dims(dims);
    if (rc != LOGO_OK) return rc;
    if ((rc = check_attn_ptrs(q, k, v)) != LOGO_OK) return rc;
    if (!pos || !cu_q || !n_sel_total || !o_c || !lse_c) return LOGO_ERR_INVALID_ARG;
    if (!aligned16(o_c)) return LOGO_ERR_UNSUPPORTED;
    if (!(scale >= 0.0f)) return LOGO_ERR_INVALID_ARG;
    if (scale == 0.0f) scale = 1.0f / sqrtf(static_cast<float>(dims.D));
    const size_t need = global_fwd_ws_layout(dims, nullptr, nullptr);
    if (!workspace || workspace_bytes < need || !aligned16(workspace)) return LOGO_ERR_WORKSPACE;
    GlobalFwdWs ws;
    global_fwd_ws_layout(dims, static_cast<char*>(workspace), &ws);
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int cap = dims.B * dims.T;
    const int row_elems = dims.Hq * dims.D;
    const int gather_grid = max(1, min(cap + kBM, device_sm_count() * 8));
    gather_rows_kernel<<<gather_grid, 256, 0, st>>>(q, pos, cu_q, n_sel_total, dims.B, dims.T, row_elems, ws.qc);
    const int n_sm = device_sm_count();
    global_schedule_kernel<<<1, 1024, 0, st>>>(pos, cu_q, dims.B, dims.Hq, n_sm, ws.tile_off, ws.unsorted, ws.sorted,
                                               ws.n_tiles, ws.next_item, ws.splits, ws.n_splits);
    if (cudaGetLastError() != cudaSuccess) return LOGO_ERR_CUDA;
    FwdParams prm{};
    if (!encode_bf16_4d(&prm.tm_q, ws.qc, dims.D, dims.Hq, static_cast<uint64_t>(cap) + kBM, 1, 64, kBM) ||
        !encode_bf16_4d(&prm.tm_k, k, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN) ||
        !encode_bf16_4d(&prm.tm_v, v, dims.D, dims.Hkv, dims.T, dims.B, 64, kBN))
        return LOGO_ERR_CUDA;
    prm.o = o_c;
    prm.lse = lse_c;
    prm.pos = pos;
    prm.tiles = ws.sorted;
    prm.n_tiles = ws.n_tiles;
    prm.next_item = ws.next_item;
    prm.o_part = ws.o_part;
    prm.m_part = ws.m_part;
    prm.l_part = ws.l_part;
    prm.B = dims.B;
    prm.T = dims.T;
    prm.Hq = dims.Hq;
    prm.Hkv = dims.Hkv;
    prm.window = kNoWindow;
    prm.cap = cap;
    prm.q_tiles = 0;
    prm.scale_log2 = scale * kLog2e;
    const int n_items_upper =
        static_cast<int>((static_cast<int64_t>(cap) / kBM + dims.B) * dims.Hq + kMaxPartialUnits);
    rc = dims.D == 128 ? launch_fwd<128, true>(prm, n_items_upper, st) : launch_fwd<64, true>(prm, n_items_upper, st);
    if (rc != LOGO_OK) return rc;
    // always launched (a fixed launch sequence, capturable in a graph); exits at once without splits
    const int merge_grid = n_sm * 4;
    if (dims.D == 128)
        merge_splits_kernel<128><<<merge_grid, 128, 0, st>>>(ws.splits, ws.n_splits, dims.Hq, cap, ws.o_part,
                                                             ws.m_part, ws.l_part, o_c, lse_c);
    else
        merge_splits_kernel<64><<<merge_grid, 128, 0, st>>>(ws.splits, ws.n_splits, dims.Hq, cap, ws.o_part,
                                                            ws.m_part, ws.l_part, o_c, lse_c);
    return cudaGetLastError() == cudaSuccess ? LOGO_OK : LOGO_ERR_CUDA;
}
