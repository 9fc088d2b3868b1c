/*
 * logo.h -- C ABI of the GB300 (sm_103a) LoGo attention hot path.
 *
 * LoGo (arXiv 2608.29539) gives every token sliding-window attention and lets
 * a per-token gate send the selected tokens' queries, in addition, to full
 * causal attention; the two normalised branch outputs are mixed by the gate.
 * This library computes that layer's data-parallel path, forward and backward:
 *
 *   logo_select                  Eq. 7 threshold / per-sequence ratio, packing of I
 *   logo_local_attn_fwd / _bwd   Eq. 6 local branch, window W, every token
 *   logo_global_sparse_attn_fwd / _bwd
 *                                Eq. 8 global branch on the selected rows only
 *   logo_combine / _bwd          Eq. 9 ContextNorm + Eq. 10 gate-weighted fusion
 *   logo_combine_bwd_gains       ... plus the gradients of the ContextNorm gains
 *   logo_gate_select / logo_gate_bwd
 *                                Eq. 7 gate p = sigmoid(x . w_g) fused ahead of
 *                                logo_select, and its backward
 *   logo_branch_transform / _bwd Eq. 5 LP / SO transforms U^L -> U^G (Q on the
 *                                selected rows only)
 *
 * Conventions shared by every entry point
 *   - All tensor pointers are DEVICE pointers owned by the caller.  The
 *     library allocates no device memory: scratch comes from a caller
 *     workspace of at least logo_*_workspace_size() bytes (16-byte aligned;
 *     256-byte alignment recommended).
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL = legacy
 *     default stream) and returns a status: LOGO_OK, or a negative LOGO_ERR_*
 *     found on the host before anything was launched (bad argument, shape the
 *     kernels do not support, launch failure).  Errors found on the device
 *     (an expired bounded wait) are reported by logo_get_device_status().
 *   - Layouts are row-major.  Q, K, V, O and their gradients are
 *     [B, T, H, D] with H = Hq for queries/outputs and H = Hkv for keys and
 *     values; bf16 tensors are passed as `logo_bf16` (raw bf16 bit patterns).
 *     Query head h reads KV head h / (Hq / Hkv) (grouped-query attention).
 *   - Positions are 0-based: token t of a sequence sees keys
 *       local : s in [max(0, t - W + 1), t]   (Sec. 3.1, C^w_t, w keys with t)
 *       global: s in [0, t]                   (Sec. 3.1, C^inf_t)
 *   - Packed ("compacted") global rows follow App. B: the selected tokens of
 *     sequence 0 in ascending position, then those of sequence 1, ...
 *     Capacity is cap = B*T rows, so no call needs the count on the host.
 *   - `scale` is the softmax temperature (Eq. 1 uses 1/sqrt(D)); pass 0 for
 *     1/sqrt(D).  Softmax statistics `lse` are natural-log log-sum-exp values
 *     of scale * q.k over the visible keys.
 *   - Supported: D in {64, 128}; Hq % Hkv == 0; T >= 1; every tensor pointer
 *     16-byte aligned and contiguous.
 */
#ifndef LOGO_H
#define LOGO_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define LOGO_API __attribute__((visibility("default")))
#else
#define LOGO_API
#endif

typedef uint16_t logo_bf16; /* bf16 bit pattern */

#define LOGO_OK 0
#define LOGO_ERR_INVALID_ARG (-1) /* null pointer, bad size, bad mode       */
#define LOGO_ERR_UNSUPPORTED (-2) /* D not 64/128, Hq % Hkv != 0, misaligned */
#define LOGO_ERR_CUDA (-3)        /* a CUDA runtime/driver call failed      */
#define LOGO_ERR_TIMEOUT (-4)     /* device: a bounded wait expired         */
#define LOGO_ERR_WORKSPACE (-5)   /* workspace missing or too small         */
#define LOGO_ERR_SCRATCH_LIMIT (-6) /* shape beyond a built-in scratch limit */

#define LOGO_SELECT_THRESHOLD 0 /* z_t = 1[p_t > b_th]                       */
#define LOGO_SELECT_RATIO 1     /* top floor(ratio*T) gates per sequence     */

typedef struct logo_dims {
    int B;   /* sequences                        */
    int T;   /* tokens per sequence              */
    int Hq;  /* query heads                      */
    int Hkv; /* key/value heads (Hq % Hkv == 0)  */
    int D;   /* head dimension (64 or 128)       */
} logo_dims;

/* Reads and clears the device error word of every kernel of the library
 * (synchronises the device).  *status receives LOGO_OK or the first
 * LOGO_ERR_* a kernel recorded since the last call.  Returns LOGO_OK, or
 * LOGO_ERR_CUDA if the word could not be read. */
LOGO_API int logo_get_device_status(int* status);

/* Number of SMs the persistent kernels size their grids for (device 0 of the
 * current context); informational. */
LOGO_API int logo_num_sms(void);

/* Self-test of the bounded device waits (no counterpart in the paper).  Every
 * pipelined kernel waits on shared-memory mbarriers with a wall-clock budget
 * (2 s); when a budget runs out the kernel records LOGO_ERR_TIMEOUT, stops its
 * roles and returns, so a lost arrival becomes a status instead of a hang.
 * This call launches one warp that waits, through that same wait, on an
 * mbarrier nothing will ever arrive at, with a budget of budget_ns
 * nanoseconds (1 .. 2e9).  After it completes, logo_get_device_status()
 * reports LOGO_ERR_TIMEOUT, and the context remains usable.  No device fault
 * or trap is involved.  Returns LOGO_ERR_INVALID_ARG for a budget out of
 * range, LOGO_ERR_CUDA if the launch fails. */
LOGO_API int logo_selftest_wait_expiry(uint64_t budget_ns, void* stream);

/* ------------------------------------------------------------------------
 * logo_select -- routing decision and packing of the selected set.
 *   Eq. 7 (Sec. 3.2): z_t = 1[p_t > b_th], the gate p_t = sigmoid(x_t . w_g)
 *   is computed by the caller; one decision per token, shared by all heads
 *   (Sec. 3.1, after Eq. 2).  I = {t : z_t = 1} (Sec. 3.2), packed as in App. B.
 *   mode LOGO_SELECT_THRESHOLD: strict float32 compare with b_th; b_th < 0
 *     selects every token (the P-mask start of Sec. 3.2), b_th >= 1 none.
 *   mode LOGO_SELECT_RATIO: in each sequence exactly k = floor(ratio * T)
 *     tokens, those with the largest p_t; equal gates go to the lower position
 *     (-0.0 and +0.0 compare equal).  ratio in [0, 1].  Gates must not be NaN.
 * In : gate_p [B,T] float32.
 * Out: z [B,T] uint8 (0/1); pos [B*T] int32 (in-sequence position of each
 *      packed row; entries >= n_sel_total are left untouched); cu_q [B+1]
 *      int32 (packed rows of sequence b are cu_q[b]..cu_q[b+1]); row_of [B,T]
 *      int32 (packed row of a selected token, -1 otherwise); n_sel_total [1]
 *      int32 (N = cu_q[B]; the realised ratio of Eq. 3 is N / (B*T)).
 * Workspace: logo_select_workspace_size(dims) bytes.
 * Integer outputs are bit-exact and deterministic. */
LOGO_API size_t logo_select_workspace_size(logo_dims dims);
LOGO_API int logo_select(const float* gate_p, logo_dims dims, int mode, float b_th, float ratio, uint8_t* z, int32_t* pos,
                int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total, void* workspace, size_t workspace_bytes,
                void* stream);

/* logo_select_device_threshold -- logo_select in LOGO_SELECT_THRESHOLD mode
 *   with the Eq. 7 threshold read by the kernels from DEVICE memory (b_th:
 *   one float32, caller-owned), so that logo_budget_update can move it
 *   between steps without a host round trip (Sec. 3.2, Budget Control).
 *   Same outputs, workspace (logo_select_workspace_size) and guarantees as
 *   logo_select in threshold mode with that value; b_th must not be written
 *   while the call runs on the stream (stream order suffices). */
LOGO_API int logo_select_device_threshold(const float* gate_p, logo_dims dims, const float* b_th, uint8_t* z,
                int32_t* pos, int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total, void* workspace,
                size_t workspace_bytes, void* stream);

/* logo_budget_update -- the budget controller of Sec. 3.2 on the device.
 *   Eq. 3: F = N / (B*T) with N = *n_sel_total (the count logo_select wrote;
 *   every token of the batch counts as valid); Eq. 11:
 *     b_th <- b_th + gamma * sign(F - rho),  sign(0) = 0,
 *   so F > rho raises the threshold (fewer tokens next step) and F < rho
 *   lowers it.  F and the sign are evaluated in double; b_th (device, one
 *   float32, updated in place) and gamma are float32 and the update is one
 *   float32 addition, so the trajectory is exact and reproducible.
 * In : n_sel_total [1] int32 (device); rho in [0, 1]; gamma >= 0 finite.
 * Out: b_th [1] float32 (device, read and written); f_out [1] float32
 *      (device, optional: F as float32; NULL to skip).
 * One single-thread launch on `stream`. */
LOGO_API int logo_budget_update(const int32_t* n_sel_total, logo_dims dims, float rho, float gamma, float* b_th,
                float* f_out, void* stream);

/* logo_pmask_initial_threshold -- P-mask start value (Sec. 3.2 Progressive
 *   Masking, App. C.1): 0.5 - gamma * pmask_steps, computed in double and
 *   returned as float32.  While every token is selected (F = 1 > rho) Eq. 11
 *   raises b_th by gamma per step, so it reaches the gate centre 0.5 when the
 *   P-mask phase of pmask_steps steps ends; until then b_th < 0 < p_t selects
 *   every token.  Host function, no device work. */
LOGO_API float logo_pmask_initial_threshold(float gamma, long long pmask_steps);

/* logo_decode_workspace_size / logo_decode_local_attn /
 * logo_decode_global_sparse_attn -- one autoregressive decoding step
 *   (Sec. 3.3 Autoregressive Decoding): each of the B sequences has one new
 *   token whose queries are q [B, Hq, D] (the local-branch queries for the
 *   local call, the global-branch queries for the global call) and
 *   seq_len[b] >= 1 tokens in its caches, the new one included, so the new
 *   token sits at position seq_len[b] - 1.  The gate and routing of the step
 *   come from logo_select (or logo_select_device_threshold) run on dims
 *   (B, T = 1), and the two outputs are fused by logo_combine on dims
 *   (B, T = 1): the same calls as in prefill.
 *   local : Eq. 6 for the new token: the keys at positions
 *           [max(0, len - W), len - 1], read from ring caches k_ring, v_ring
 *           [B, R, Hkv, D] with R = dims.T >= W slots, position s in slot
 *           s mod R.  Out: o [B, Hq, D].
 *   global: Eq. 8 for the selected sequences only: packed row r (the r-th
 *           selected sequence b, ascending; cu_q [B+1] and n_sel_total [1]
 *           from the selection, device) attends positions [0, len - 1] of its
 *           dense caches k_cache, v_cache [B, L, Hkv, D], L = dims.T >= len.
 *           Out: o_c [B, Hq, D], packed rows; rows >= n_sel_total are left
 *           untouched.  The work of unselected sequences is never launched
 *           (the device-side count bounds it), so they read none of their
 *           cache (the compaction the paper names as the missing serving
 *           kernel) and no host synchronisation is needed.
 *   Cache rows the step does not see (past seq_len, outside the window) may
 *   hold anything.  dims: B, T = R or L, Hq, Hkv (Hq / Hkv <= 16), D in
 *   {64, 128}; window >= 1 (local); scale as elsewhere (0 = 1/sqrt(D)).
 *   Workspace: logo_decode_workspace_size(dims) bytes (per-chunk fp32
 *   partials), one workspace per call in flight. */
LOGO_API size_t logo_decode_workspace_size(logo_dims dims);
LOGO_API int logo_decode_local_attn(const logo_bf16* q, const logo_bf16* k_ring, const logo_bf16* v_ring,
                const int32_t* seq_len, logo_bf16* o, logo_dims dims, int window, float scale, void* workspace,
                size_t workspace_bytes, void* stream);
LOGO_API int logo_decode_global_sparse_attn(const logo_bf16* q, const logo_bf16* k_cache, const logo_bf16* v_cache,
                const int32_t* seq_len, const int32_t* cu_q, const int32_t* n_sel_total, logo_bf16* o_c,
                logo_dims dims, float scale, void* workspace, size_t workspace_bytes, void* stream);

/* logo_select_noalloc -- logo_select for callers that cannot allocate.
 *   No counterpart in the paper: this is a deployment variant of logo_select.
 *   Some callers hold only their own input and output buffers and have no way
 *   to obtain a workspace: a serving runtime that fixes all device memory
 *   when it starts and forbids allocation per request, or a host in another
 *   language that reaches this library through a plain C FFI without any
 *   CUDA allocator of its own.  This entry point takes the same inputs and
 *   outputs as logo_select (same results, bit for bit) and no workspace: its
 *   scratch is a static device array of LOGO_SELECT_NOALLOC_SCRATCH_BYTES
 *   inside the library, which every GPU that loads the library holds until the
 *   process exits.  It calls no cudaMalloc, cudaFree or allocating routine.
 *   Limits: B <= LOGO_SELECT_NOALLOC_MAX_SEQS and B * ceil(T / 1024) <=
 *   LOGO_SELECT_NOALLOC_MAX_CHUNKS (at most 16,777,216 tokens per call);
 *   larger shapes return LOGO_ERR_SCRATCH_LIMIT before anything is launched.
 *   The first call in each CUDA context looks up the array's device address
 *   (cudaGetSymbolAddress, with that device current) and caches it under the
 *   context's id: make that first call before any stream capture, and again
 *   after anything that recreates the context (cudaDeviceReset), which the
 *   next call notices and repeats the lookup for.  All calls share the one array, which keeps
 *   the previous call's contents; every kernel writes the scratch it reads
 *   before reading it, so no clearing is needed, but calls that overlap on
 *   the GPU (different streams, or concurrent host threads) race on it and
 *   must be serialised by the caller. */
#define LOGO_SELECT_NOALLOC_MAX_SEQS 4096
#define LOGO_SELECT_NOALLOC_MAX_CHUNKS 16384
#define LOGO_SELECT_NOALLOC_SCRATCH_BYTES 294912
LOGO_API int logo_select_noalloc(const float* gate_p, logo_dims dims, int mode, float b_th, float ratio, uint8_t* z,
                                 int32_t* pos, int32_t* cu_q, int32_t* row_of, int32_t* n_sel_total, void* stream);

/* ------------------------------------------------------------------------
 * logo_local_attn_fwd -- local branch O^L = SoftmaxAttn_W(Q^L, K^L, V^L)
 *   (Eq. 6 with Eq. 1 over C^w_t), for all B*T tokens.  window >= 1;
 *   window >= T is full causal attention.
 * In : q [B,T,Hq,D], k/v [B,T,Hkv,D] bf16.
 * Out: o [B,T,Hq,D] bf16; lse [B,Hq,T] float32 (kept for the backward).
 * bf16 MMA on tcgen05 tensor cores with fp32 accumulation and softmax. */
LOGO_API int logo_local_attn_fwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, logo_bf16* o, float* lse,
                        logo_dims dims, int window, float scale, void* stream);

/* logo_local_attn_bwd -- gradients of logo_local_attn_fwd.
 * In : q, k, v, o, lse as in/out of the forward; dO [B,T,Hq,D] bf16.
 * Out: dq [B,T,Hq,D], dk/dv [B,T,Hkv,D] bf16 (overwritten; dk/dv sum over
 *      the query heads of each group).
 * Workspace: logo_local_attn_bwd_workspace_size(dims) bytes (fp32 dQ
 * accumulator and row statistics). */
LOGO_API size_t logo_local_attn_bwd_workspace_size(logo_dims dims);
LOGO_API int logo_local_attn_bwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, const logo_bf16* o,
                        const float* lse, const logo_bf16* dO, logo_bf16* dq, logo_bf16* dk, logo_bf16* dv,
                        logo_dims dims, int window, float scale, void* workspace, size_t workspace_bytes,
                        void* stream);

/* ------------------------------------------------------------------------
 * logo_global_sparse_attn_fwd -- query-sparse global branch
 *   O^G_I = SoftmaxAttn_inf(Q^G_I, K^G, V^G) (Eq. 8): only the packed
 *   selected rows are computed, each against the dense causal prefix of its
 *   real position (App. B), so every selected row gets exactly the dense
 *   full-causal result.
 * In : q [B,T,Hq,D] bf16 DENSE (rows gathered by pos inside the call);
 *      k/v [B,T,Hkv,D] bf16; pos, cu_q, n_sel_total from logo_select.
 * Out: o_c [B*T, Hq, D] bf16 packed (rows >= n_sel_total untouched);
 *      lse_c [Hq, B*T] float32 packed.
 * Workspace: logo_global_attn_fwd_workspace_size(dims) bytes (packed Q and
 * the tile schedule). */
LOGO_API size_t logo_global_attn_fwd_workspace_size(logo_dims dims);
LOGO_API int logo_global_sparse_attn_fwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, const int32_t* pos,
                                const int32_t* cu_q, const int32_t* n_sel_total, logo_bf16* o_c, float* lse_c,
                                logo_dims dims, float scale, void* workspace, size_t workspace_bytes,
                                void* stream);

/* logo_global_sparse_attn_bwd -- row-sparse backward of the global branch
 *   (Sec. 3.3 and App. B): dQ only for selected rows, scattered to the dense
 *   layout with zero rows for unselected tokens; dK/dV accumulate over the
 *   selected rows that can see each key.
 * In : q, k, v, pos, cu_q, n_sel_total as in the forward; o_c, lse_c from the
 *      forward; dO_c [B*T, Hq, D] bf16 packed (rows < n_sel_total read).
 * Out: dq [B,T,Hq,D] bf16 dense (zeros on unselected rows); dk/dv
 *      [B,T,Hkv,D] bf16 (overwritten).
 * Workspace: logo_global_attn_bwd_workspace_size(dims) bytes. */
LOGO_API size_t logo_global_attn_bwd_workspace_size(logo_dims dims);
LOGO_API int logo_global_sparse_attn_bwd(const logo_bf16* q, const logo_bf16* k, const logo_bf16* v, const int32_t* pos,
                                const int32_t* cu_q, const int32_t* n_sel_total, const logo_bf16* o_c,
                                const float* lse_c, const logo_bf16* dO_c, logo_bf16* dq, logo_bf16* dk,
                                logo_bf16* dv, logo_dims dims, float scale, void* workspace,
                                size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * logo_gate_select -- the token gate of Eq. 7, p_t = sigmoid(x_t . w_g), then
 *   logo_select on p: the gate and the selection in one call.
 * In : x [B,T,d_model] bf16 (the layer input; rows contiguous, 16-byte
 *      aligned); w_g [d_model] float32 (16-byte aligned); d_model a multiple
 *      of 8 and at most 8192; mode / b_th / ratio as logo_select.  Only dims.B
 *      and dims.T are read.
 * Out: gate_p [B,T] float32: the p the selection compared (fp32 dot product
 *      over d_model, fp32 sigmoid); z, pos, cu_q, row_of, n_sel_total as
 *      logo_select.
 * Workspace: logo_select_workspace_size(dims) bytes.
 * Errors: as logo_select; LOGO_ERR_UNSUPPORTED for d_model or alignment. */
LOGO_API int logo_gate_select(const logo_bf16* x, const float* w_g, int d_model, logo_dims dims, int mode,
                              float b_th, float ratio, float* gate_p, uint8_t* z, int32_t* pos, int32_t* cu_q,
                              int32_t* row_of, int32_t* n_sel_total, void* workspace, size_t workspace_bytes,
                              void* stream);

/* logo_gate_bwd -- backward of the gate with the selection held fixed (z
 *   passes no gradient): dlogit_t = dp_t p_t (1 - p_t), dx_t = dlogit_t w_g,
 *   dw_g = sum over t of dlogit_t x_t.
 * In : x, w_g, d_model as logo_gate_select; gate_p [B,T] float32 (its
 *      output); dgate_p [B,T] float32 (e.g. from logo_combine_bwd).
 * Out: dx [B,T,d_model] bf16: written, or added to when accumulate = 1 (the
 *      caller's gradient of x from its other uses); may be NULL.  dw_g
 *      [d_model] float32, overwritten; may be NULL (not both).  dw_g is summed
 *      per block, then over the blocks in a fixed order (deterministic).
 * Workspace: logo_gate_bwd_workspace_size(dims, d_model) bytes when dw_g is
 *      requested (else may be NULL). */
LOGO_API size_t logo_gate_bwd_workspace_size(logo_dims dims, int d_model);
LOGO_API int logo_gate_bwd(const logo_bf16* x, const float* w_g, const float* gate_p, const float* dgate_p,
                           int d_model, logo_dims dims, logo_bf16* dx, int accumulate, float* dw_g, void* workspace,
                           size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * logo_branch_transform -- the per-head branch transform of Eq. 5 that turns a
 *   local-branch tensor into the global branch's, in one of its two forms:
 *   LP: U^G_h = U^L_h A_h, A [H,D,D] bf16 (A[h][i][j] maps input dimension i to
 *       output j; identity at initialisation; the paper's default);
 *   SO: U^G_h = U^L_h * s_h + b_h, s and b [H,D] float32.
 *   Exactly one form: a_lp, or both s_so and b_so.
 * Rows: every row when pos is NULL (K and V); otherwise only the packed
 *   selected rows described by pos / cu_q / n_sel_total (device, from
 *   logo_select): Q, of which the global branch reads those rows alone.
 * In : u_l [B,T,H,D] bf16 with H = dims.Hq, the head count of this tensor (Hq
 *      for Q, Hkv for K and V; dims.Hkv is not read); D 64 or 128; H*D <= 8192.
 *      LP runs on the tensor cores (warp-level MMA), SO elementwise.
 * Out: u_g [B,T,H,D] bf16: the listed rows written, other rows untouched.
 * Errors: LOGO_ERR_INVALID_ARG for a missing or doubled form or pointer;
 *      LOGO_ERR_UNSUPPORTED for D, H*D or 16-byte alignment. */
LOGO_API int logo_branch_transform(const logo_bf16* u_l, const logo_bf16* a_lp, const float* s_so, const float* b_so,
                                   const int32_t* pos, const int32_t* cu_q, const int32_t* n_sel_total,
                                   logo_bf16* u_g, logo_dims dims, void* stream);

/* logo_branch_transform_bwd -- gradients of logo_branch_transform on the same
 *   rows, for du_g [B,T,H,D] bf16 (read on the listed rows):
 *   du_l = du_g A_h^T (LP) or du_g * s_h (SO), written, or added to du_l when
 *      accumulate = 1 (the caller's gradient of U^L from the local branch);
 *   LP: da_lp [H,D,D] float32 = sum over the rows of u_l^T du_g;
 *   SO: ds_so, db_so [H,D] float32 = sums of du_g * u_l and of du_g (either may
 *      be NULL).  Parameter gradients are summed per block, then over the blocks
 *      in a fixed order (deterministic).
 * Workspace: logo_branch_transform_bwd_workspace_size(dims) bytes. */
LOGO_API size_t logo_branch_transform_bwd_workspace_size(logo_dims dims);
LOGO_API int logo_branch_transform_bwd(const logo_bf16* u_l, const logo_bf16* a_lp, const float* s_so,
                                       const int32_t* pos, const int32_t* cu_q, const int32_t* n_sel_total,
                                       const logo_bf16* du_g, logo_bf16* du_l, int accumulate, float* da_lp,
                                       float* ds_so, float* db_so, logo_dims dims, void* workspace,
                                       size_t workspace_bytes, void* stream);

/* ------------------------------------------------------------------------
 * logo_combine -- ContextNorm per branch (Eq. 9: head-wise RMSNorm over D,
 *   r = 1/sqrt(mean_d o^2 + eps), o~ = o * r * gain) and the output fusion
 *   (Eq. 10): o_t = (1 - p_t) o~L_t + p_t o~G_t if z_t = 1, else o~L_t.
 * In : o_l [B,T,Hq,D] bf16; o_c [B*T,Hq,D] bf16 packed global rows; gate_p
 *      [B,T] float32; z [B,T] uint8; row_of [B,T] int32; gain_l / gain_g
 *      [Hq,D] float32 or NULL (= 1); eps > 0.
 * Out: o [B,T,Hq,D] bf16; rstd_l [B,T,Hq] and rstd_g [B*T,Hq] float32 (the
 *      RMS reciprocals r; either may be NULL).
 * Errors: LOGO_ERR_UNSUPPORTED if D is not 64 or 128, Hq*D > 16384, or a
 *      bf16 / gain pointer is not 16-byte aligned. */
LOGO_API int logo_combine(const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p, const uint8_t* z,
                 const int32_t* row_of, const float* gain_l, const float* gain_g, float eps, logo_bf16* o,
                 float* rstd_l, float* rstd_g, logo_dims dims, void* stream);

/* logo_combine_bwd -- backward of logo_combine with z held fixed (z is a hard
 *   indicator and passes no gradient):
 *   do~L = dO (1 - p z), do~G = dO p, RMSNorm backward per branch, and
 *   dp_t = z_t * sum_{h,d} dO (o~G - o~L).
 * Out: dO_l [B,T,Hq,D] bf16; dO_c [B*T,Hq,D] bf16 packed (selected rows
 *      written); dgate_p [B,T] float32 (0 on unselected tokens). */
LOGO_API int logo_combine_bwd(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c, const float* gate_p,
                     const uint8_t* z, const int32_t* row_of, const float* gain_l, const float* gain_g, float eps,
                     logo_bf16* dO_l, logo_bf16* dO_c, float* dgate_p, logo_dims dims, void* stream);

/* logo_combine_bwd_gains -- logo_combine_bwd plus the gradients of the two
 *   ContextNorm gains (Eq. 9; o~ = o r gain is linear in the gain), z fixed:
 *   dgain_l[h,d] = sum over every token of dy^L o^L r^L, dy^L = dO (1 - p z);
 *   dgain_g[h,d] = sum over the selected tokens of dy^G o^G r^G, dy^G = dO p.
 * Out: as logo_combine_bwd, plus dgain_l / dgain_g [Hq,D] float32 (overwritten;
 *      either may be NULL, not both).  Tokens are summed per block, then the
 *      blocks in a fixed order: the result is deterministic on a given GPU.
 * Workspace: logo_combine_bwd_workspace_size(dims) bytes of device memory.
 * Errors: LOGO_ERR_UNSUPPORTED if Hq*D > 8192; LOGO_ERR_WORKSPACE if the
 *      workspace is short; otherwise as logo_combine_bwd. */
LOGO_API size_t logo_combine_bwd_workspace_size(logo_dims dims);
LOGO_API int logo_combine_bwd_gains(const logo_bf16* dO, const logo_bf16* o_l, const logo_bf16* o_c,
                                    const float* gate_p, const uint8_t* z, const int32_t* row_of,
                                    const float* gain_l, const float* gain_g, float eps, logo_bf16* dO_l,
                                    logo_bf16* dO_c, float* dgate_p, float* dgain_l, float* dgain_g,
                                    logo_dims dims, void* workspace, size_t workspace_bytes, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* LOGO_H */
