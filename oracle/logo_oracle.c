/*
 * logo_oracle.c -- plain, slow, obviously-correct CPU reference of the LoGo
 * attention layer's data-parallel hot path (arXiv 2608.29539, Sec. 3.2-3.3).
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call this code:
 * only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference
 * arm use it.  It shares no code, header, table or helper with the CUDA path.
 *
 * Arithmetic is IEEE double throughout (the paper fixes no precision); inputs
 * arrive as float32 arrays holding exactly the values the GPU receives
 * (bf16-rounded where the GPU takes bf16).  The only decisions made in float32
 * are the gate comparisons of Eq. 7, which the GPU makes in float32 too.
 *
 * Conventions (0-based positions; the paper writes 1-based):
 *   Q, K, V       [B, T, H, D] row-major (Hq query heads, Hkv key/value heads)
 *   local window  keys s in [max(0, t-W+1), t]            (Sec. 3.1, C^w_t)
 *   global        keys s in [0, t]                          (Sec. 3.1, C^inf_t)
 *   GQA           query head h reads KV head h / (Hq/Hkv)
 *
 * parity pins: every function here is pinned by tests/test_oracle_pins.py
 * (library routines, closed forms, finite differences, special cases).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ------------------------------------------------------------------------ */
/* Eq. 7: z_t = 1[p_t > b_th], strict comparison, float32 operands.          */
/* ------------------------------------------------------------------------ */
void oracle_select_threshold(const float* p, int64_t n, float b_th, uint8_t* z)
{
    for (int64_t i = 0; i < n; ++i) z[i] = (p[i] > b_th) ? 1 : 0;
}

/* Eq. 7 gate: p_t = sigmoid(x_t . w_g) in double, x [N, dm] (float32 holding
 * the bf16 values the GPU reads), w_g [dm]. */
void oracle_gate(const float* x, const float* w, int64_t n, int dm, double* p)
{
    for (int64_t t = 0; t < n; ++t) {
        double a = 0.0;
        for (int i = 0; i < dm; ++i) a += (double)x[t * dm + i] * (double)w[i];
        p[t] = 1.0 / (1.0 + exp(-a));
    }
}

/* Backward of oracle_gate for a given dp: with p recomputed in double,
 * dlogit_t = dp_t p_t (1 - p_t) (the sigmoid's derivative),
 * dx_t = dlogit_t w_g, dw_g = sum over t (in order) of dlogit_t x_t. */
void oracle_gate_bwd(const float* x, const float* w, const float* dp, int64_t n, int dm, double* dx, double* dw)
{
    memset(dw, 0, sizeof(double) * (size_t)dm);
    for (int64_t t = 0; t < n; ++t) {
        double a = 0.0;
        for (int i = 0; i < dm; ++i) a += (double)x[t * dm + i] * (double)w[i];
        double pt = 1.0 / (1.0 + exp(-a));
        double g = (double)dp[t] * pt * (1.0 - pt);
        for (int i = 0; i < dm; ++i) {
            dx[t * dm + i] = g * (double)w[i];
            dw[i] += g * (double)x[t * dm + i];
        }
    }
}

/* Eq. 5 branch transform U^G_h = phi_{U,h}(U^L_h), for the listed rows r
 * (indices into the B*T rows of a [B,T,H,D] tensor), in double:
 *   LP (A != NULL): g[r,h,j] = sum_i u[r,h,i] A[h,i,j]      A [H,D,D]
 *   SO (A == NULL): g[r,h,j] = u[r,h,j] s[h,j] + b[h,j]      s, b [H,D]
 * Output g [nrows,H,D]. */
void oracle_branch_fwd(const float* u, int H, int D, const int64_t* rows, int64_t nrows, const float* A,
                       const float* s, const float* b, double* g)
{
    for (int64_t r = 0; r < nrows; ++r) {
        for (int h = 0; h < H; ++h) {
            const float* ur = u + (rows[r] * H + h) * (int64_t)D;
            double* gr = g + (r * H + h) * (int64_t)D;
            for (int j = 0; j < D; ++j) {
                if (A) {
                    double acc = 0.0;
                    for (int i = 0; i < D; ++i) acc += (double)ur[i] * (double)A[((int64_t)h * D + i) * D + j];
                    gr[j] = acc;
                } else {
                    gr[j] = (double)ur[j] * (double)s[(int64_t)h * D + j] + (double)b[(int64_t)h * D + j];
                }
            }
        }
    }
}

/* Gradients of oracle_branch_fwd for dg [nrows,H,D]:
 *   LP: du[r,h,i] = sum_j dg[r,h,j] A[h,i,j];  dA[h,i,j] = sum_r u[r,h,i] dg[r,h,j]
 *   SO: du = dg s;  ds[h,j] = sum_r dg u;  db[h,j] = sum_r dg
 * Parameter gradients summed over the rows in order. */
void oracle_branch_bwd(const float* u, int H, int D, const int64_t* rows, int64_t nrows, const float* A,
                       const float* s, const float* dg, double* du, double* dA, double* ds, double* db)
{
    if (A) memset(dA, 0, sizeof(double) * (size_t)H * D * D);
    else {
        memset(ds, 0, sizeof(double) * (size_t)H * D);
        memset(db, 0, sizeof(double) * (size_t)H * D);
    }
    for (int64_t r = 0; r < nrows; ++r) {
        for (int h = 0; h < H; ++h) {
            const float* ur = u + (rows[r] * H + h) * (int64_t)D;
            const float* gr = dg + (r * H + h) * (int64_t)D;
            double* dur = du + (r * H + h) * (int64_t)D;
            for (int i = 0; i < D; ++i) {
                if (A) {
                    double acc = 0.0;
                    for (int j = 0; j < D; ++j) acc += (double)gr[j] * (double)A[((int64_t)h * D + i) * D + j];
                    dur[i] = acc;
                    for (int j = 0; j < D; ++j) dA[((int64_t)h * D + i) * D + j] += (double)ur[i] * (double)gr[j];
                } else {
                    dur[i] = (double)gr[i] * (double)s[(int64_t)h * D + i];
                    ds[(int64_t)h * D + i] += (double)gr[i] * (double)ur[i];
                    db[(int64_t)h * D + i] += (double)gr[i];
                }
            }
        }
    }
}

/* Eq. 3 and Eq. 11 (Sec. 3.2, Budget Control): the realised ratio is
 * F = n_sel / n_valid, and the threshold moves by gamma * sign(F - rho).
 * F and the sign are evaluated in double from the integer counts; b_th and
 * gamma are float32 (the precision of the gate and of the Eq. 7 compare) and
 * the update is one float32 addition.  Returns the new b_th; *F_out = F. */
float oracle_budget_update(int64_t n_sel, int64_t n_valid, float rho, float gamma, float b_th, double* F_out)
{
    const double F = (double)n_sel / (double)n_valid;
    const double d = F - (double)rho;
    const float sgn = d > 0.0 ? 1.0f : (d < 0.0 ? -1.0f : 0.0f);
    const float step = gamma * sgn; /* exact: sgn is -1, 0 or +1 */
    if (F_out) *F_out = F;
    return b_th + step;
}

/* P-mask start (Sec. 3.2 Progressive Masking, App. C.1): b_th starts at the
 * gate centre 0.5 minus the total drift of S steps at rate gamma, so that
 * while every token is selected (F = 1 > rho) it reaches 0.5 after S steps.
 * Computed in double. */
double oracle_pmask_threshold(double gamma, int64_t steps) { return 0.5 - gamma * (double)steps; }

/* Ratio mode: in each sequence the k tokens with the largest gate p_t are
 * selected; equal gates are ordered by lower position first.  This is the
 * per-sequence quantile reading of the target ratio rho (k = floor(rho*T)),
 * computed here by a full sort of (p descending, t ascending). */
static const float* g_sort_p;
static int cmp_desc_p_then_t(const void* a, const void* b)
{
    int ia = *(const int*)a, ib = *(const int*)b;
    float pa = g_sort_p[ia], pb = g_sort_p[ib];
    if (pa > pb) return -1;
    if (pa < pb) return 1;
    return (ia < ib) ? -1 : (ia > ib);
}

void oracle_select_ratio(const float* p, int B, int T, int k, uint8_t* z)
{
    int* idx = (int*)malloc(sizeof(int) * (size_t)(T > 0 ? T : 1));
    for (int b = 0; b < B; ++b) {
        const float* pb = p + (int64_t)b * T;
        uint8_t* zb = z + (int64_t)b * T;
        for (int t = 0; t < T; ++t) { idx[t] = t; zb[t] = 0; }
        g_sort_p = pb;
        qsort(idx, (size_t)T, sizeof(int), cmp_desc_p_then_t);
        for (int i = 0; i < k && i < T; ++i) zb[idx[i]] = 1;
    }
    free(idx);
}

/* Selected set I = {t : z_t = 1} (Sec. 3.2), packed in ascending position
 * order per sequence, sequences one after another (App. B): pos[] holds the
 * in-sequence position of each packed row, cu_q[b]..cu_q[b+1] the rows of
 * sequence b, row_of[b,t] the packed row of token (b,t) or -1.
 * Returns N = total number of selected tokens (numerator of Eq. 3). */
int64_t oracle_compact(const uint8_t* z, int B, int T, int32_t* pos, int32_t* cu_q, int32_t* row_of)
{
    int64_t n = 0;
    for (int b = 0; b < B; ++b) {
        cu_q[b] = (int32_t)n;
        for (int t = 0; t < T; ++t) {
            int64_t bt = (int64_t)b * T + t;
            if (z[bt]) { pos[n] = t; row_of[bt] = (int32_t)n; ++n; }
            else row_of[bt] = -1;
        }
    }
    cu_q[B] = (int32_t)n;
    return n;
}

/* ------------------------------------------------------------------------ */
/* Eq. 1 softmax attention for a list of query rows.                          */
/* ------------------------------------------------------------------------ */
static inline int64_t idx4(int b, int t, int h, int T, int H, int D)
{
    return (((int64_t)b * T + t) * H + h) * (int64_t)D;
}

/* Visible keys of query position t: window > 0 gives C^w_t, window <= 0 C^inf_t. */
static inline int key_lo(int t, int window) { return (window > 0 && t - window + 1 > 0) ? t - window + 1 : 0; }

/* Forward.  Row r is query (row_b[r], row_t[r]); for every listed head h:
 *   l_s   = scale * q_t . k_s            s in C_t
 *   o_t   = sum_s softmax(l)_s v_s        (Eq. 1)
 *   lse_t = log sum_s exp(l_s)            (natural log)
 * o: [nrows, Hq, D], lse: [nrows, Hq]; entries of heads not listed are left
 * untouched. */
void oracle_attn_fwd(const float* q, const float* k, const float* v,
                     int B, int T, int Hq, int Hkv, int D,
                     int64_t nrows, const int32_t* row_b, const int32_t* row_t,
                     int nheads, const int32_t* heads,
                     int window, double scale, double* o, double* lse)
{
    (void)B;
    const int group = Hq / Hkv;
    int64_t total = nrows * (int64_t)nheads;
#pragma omp parallel
    {
        double* l = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
#pragma omp for schedule(dynamic, 16)
        for (int64_t w = 0; w < total; ++w) {
            int64_t r = w / nheads;
            int h = heads[w % nheads];
            int b = row_b[r], t = row_t[r];
            int kvh = h / group;
            int lo = key_lo(t, window);
            const float* qr = q + idx4(b, t, h, T, Hq, D);
            double m = -INFINITY;
            for (int s = lo; s <= t; ++s) {
                const float* ks = k + idx4(b, s, kvh, T, Hkv, D);
                double acc = 0.0;
                for (int d = 0; d < D; ++d) acc += (double)qr[d] * (double)ks[d];
                l[s - lo] = acc * scale;
                if (l[s - lo] > m) m = l[s - lo];
            }
            double sum = 0.0;
            for (int s = lo; s <= t; ++s) { l[s - lo] = exp(l[s - lo] - m); sum += l[s - lo]; }
            double* orow = o + (r * Hq + h) * (int64_t)D;
            for (int d = 0; d < D; ++d) orow[d] = 0.0;
            for (int s = lo; s <= t; ++s) {
                const float* vs = v + idx4(b, s, kvh, T, Hkv, D);
                double a = l[s - lo] / sum;
                for (int d = 0; d < D; ++d) orow[d] += a * (double)vs[d];
            }
            lse[r * Hq + h] = m + log(sum);
        }
        free(l);
    }
}

/* Backward of the same operator with the row set held fixed (z is a hard
 * indicator and carries no gradient).  With P = softmax(l) over C_t and the
 * upstream gradient dO of row t:
 *   dP_s = dO_t . v_s
 *   dl_s = P_s (dP_s - sum_j P_j dP_j)          (softmax Jacobian)
 *   dq_t += scale * sum_s dl_s k_s
 *   dk_s += scale * dl_s q_t ,   dv_s += P_s dO_t
 * dO: [nrows, Hq, D]; dq: [nrows, Hq, D]; dk, dv: [B, T, Hkv, D] (must be
 * zeroed by the caller; KV heads accumulate over the listed query heads of
 * their group, so list whole groups to get the full dK/dV). */
void oracle_attn_bwd(const float* q, const float* k, const float* v,
                     int B, int T, int Hq, int Hkv, int D,
                     int64_t nrows, const int32_t* row_b, const int32_t* row_t,
                     int nheads, const int32_t* heads,
                     int window, double scale, const float* dO,
                     double* dq, double* dk, double* dv)
{
    const int group = Hq / Hkv;
    int64_t total = (int64_t)B * Hkv;
#pragma omp parallel
    {
        double* P = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
        double* dP = (double*)malloc(sizeof(double) * (size_t)(T > 0 ? T : 1));
#pragma omp for schedule(dynamic, 1)
        for (int64_t w = 0; w < total; ++w) {
            int b = (int)(w / Hkv), kvh = (int)(w % Hkv);
            for (int hi = 0; hi < nheads; ++hi) {
                int h = heads[hi];
                if (h / group != kvh) continue;
                for (int64_t r = 0; r < nrows; ++r) {
                    if (row_b[r] != b) continue;
                    int t = row_t[r];
                    int lo = key_lo(t, window);
                    const float* qr = q + idx4(b, t, h, T, Hq, D);
                    const float* dor = dO + (r * Hq + h) * (int64_t)D;
                    double m = -INFINITY;
                    for (int s = lo; s <= t; ++s) {
                        const float* ks = k + idx4(b, s, kvh, T, Hkv, D);
                        double acc = 0.0;
                        for (int d = 0; d < D; ++d) acc += (double)qr[d] * (double)ks[d];
                        P[s - lo] = acc * scale;
                        if (P[s - lo] > m) m = P[s - lo];
                    }
                    double sum = 0.0;
                    for (int s = lo; s <= t; ++s) { P[s - lo] = exp(P[s - lo] - m); sum += P[s - lo]; }
                    double pdp = 0.0;
                    for (int s = lo; s <= t; ++s) {
                        P[s - lo] /= sum;
                        const float* vs = v + idx4(b, s, kvh, T, Hkv, D);
                        double acc = 0.0;
                        for (int d = 0; d < D; ++d) acc += (double)dor[d] * (double)vs[d];
                        dP[s - lo] = acc;
                        pdp += P[s - lo] * acc;
                    }
                    double* dqr = dq + (r * Hq + h) * (int64_t)D;
                    for (int d = 0; d < D; ++d) dqr[d] = 0.0;
                    for (int s = lo; s <= t; ++s) {
                        double ds = P[s - lo] * (dP[s - lo] - pdp);
                        const float* ks = k + idx4(b, s, kvh, T, Hkv, D);
                        double* dks = dk + idx4(b, s, kvh, T, Hkv, D);
                        double* dvs = dv + idx4(b, s, kvh, T, Hkv, D);
                        for (int d = 0; d < D; ++d) {
                            dqr[d] += scale * ds * (double)ks[d];
                            dks[d] += scale * ds * (double)qr[d];
                            dvs[d] += P[s - lo] * (double)dor[d];
                        }
                    }
                }
            }
        }
        free(P);
        free(dP);
    }
}

/* ------------------------------------------------------------------------ */
/* Eq. 9 ContextNorm (head-wise RMSNorm over d) and Eq. 10 output fusion.     */
/* ------------------------------------------------------------------------ */
/* r = 1/sqrt(mean_d x^2 + eps); y_d = x_d * r * g_d  (g == NULL means 1). */
static double rms_fwd(const float* x, const float* g, double eps, int D, double* y)
{
    double ss = 0.0;
    for (int d = 0; d < D; ++d) ss += (double)x[d] * (double)x[d];
    double r = 1.0 / sqrt(ss / D + eps);
    for (int d = 0; d < D; ++d) y[d] = (double)x[d] * r * (g ? (double)g[d] : 1.0);
    return r;
}

/* Given dy for y = rms_fwd(x): dx_j = r g_j dy_j - x_j r^3 mean_d(x_d g_d dy_d). */
static void rms_bwd(const float* x, const float* g, double eps, int D, const double* dy, double* dx)
{
    double ss = 0.0, xgdy = 0.0;
    for (int d = 0; d < D; ++d) {
        ss += (double)x[d] * (double)x[d];
        xgdy += (double)x[d] * (g ? (double)g[d] : 1.0) * dy[d];
    }
    double r = 1.0 / sqrt(ss / D + eps);
    for (int d = 0; d < D; ++d)
        dx[d] = r * (g ? (double)g[d] : 1.0) * dy[d] - (double)x[d] * r * r * r * xgdy / D;
}

/* Fusion (Eq. 10): o_t = (1-p_t) oL~_t + p_t oG~_t if z_t = 1, else oL~_t,
 * with oL~ = Norm^L(O^L), oG~ = Norm^G(O^G) (Eq. 9).
 * oL: [B,T,H,D]; oGc: [N,H,D] packed global rows (row_of maps token -> row);
 * gL, gG: [H,D] or NULL.  Outputs o [B,T,H,D], rstdL [B,T,H], rstdG [N,H]. */
void oracle_combine_fwd(const float* oL, const float* oGc, const float* p, const uint8_t* z,
                        const int32_t* row_of, const float* gL, const float* gG, double eps,
                        int B, int T, int H, int D, double* o, double* rstdL, double* rstdG)
{
    int64_t ntok = (int64_t)B * T;
#pragma omp parallel
    {
        double* yl = (double*)malloc(sizeof(double) * (size_t)D);
        double* yg = (double*)malloc(sizeof(double) * (size_t)D);
#pragma omp for schedule(static)
        for (int64_t bt = 0; bt < ntok; ++bt) {
            for (int h = 0; h < H; ++h) {
                const float* xl = oL + (bt * H + h) * (int64_t)D;
                double* orow = o + (bt * H + h) * (int64_t)D;
                rstdL[bt * H + h] = rms_fwd(xl, gL ? gL + (int64_t)h * D : NULL, eps, D, yl);
                if (z[bt]) {
                    int64_t row = row_of[bt];
                    const float* xg = oGc + (row * H + h) * (int64_t)D;
                    rstdG[row * H + h] = rms_fwd(xg, gG ? gG + (int64_t)h * D : NULL, eps, D, yg);
                    double pt = (double)p[bt];
                    for (int d = 0; d < D; ++d) orow[d] = (1.0 - pt) * yl[d] + pt * yg[d];
                } else {
                    for (int d = 0; d < D; ++d) orow[d] = yl[d];
                }
            }
        }
        free(yl);
        free(yg);
    }
}

/* Backward of the fusion with z held fixed:
 *   doL~ = dO * (z ? 1-p : 1),  doG~ = dO * p (selected rows only)
 *   dO^L, dO^G from the RMSNorm backward,
 *   dp_t = z_t * sum_{h,d} dO (oG~ - oL~).
 * dOL: [B,T,H,D]; dOGc: [N,H,D]; dp: [B,T]. */
void oracle_combine_bwd(const float* dO, const float* oL, const float* oGc, const float* p,
                        const uint8_t* z, const int32_t* row_of, const float* gL, const float* gG,
                        double eps, int B, int T, int H, int D,
                        double* dOL, double* dOGc, double* dp)
{
    int64_t ntok = (int64_t)B * T;
#pragma omp parallel
    {
        double* yl = (double*)malloc(sizeof(double) * (size_t)D);
        double* yg = (double*)malloc(sizeof(double) * (size_t)D);
        double* dy = (double*)malloc(sizeof(double) * (size_t)D);
#pragma omp for schedule(static)
        for (int64_t bt = 0; bt < ntok; ++bt) {
            double pt = (double)p[bt];
            double acc = 0.0;
            for (int h = 0; h < H; ++h) {
                const float* g = dO + (bt * H + h) * (int64_t)D;
                const float* xl = oL + (bt * H + h) * (int64_t)D;
                const float* gl = gL ? gL + (int64_t)h * D : NULL;
                double wl = z[bt] ? 1.0 - pt : 1.0;
                for (int d = 0; d < D; ++d) dy[d] = (double)g[d] * wl;
                rms_bwd(xl, gl, eps, D, dy, dOL + (bt * H + h) * (int64_t)D);
                if (z[bt]) {
                    int64_t row = row_of[bt];
                    const float* xg = oGc + (row * H + h) * (int64_t)D;
                    const float* gg = gG ? gG + (int64_t)h * D : NULL;
                    for (int d = 0; d < D; ++d) dy[d] = (double)g[d] * pt;
                    rms_bwd(xg, gg, eps, D, dy, dOGc + (row * H + h) * (int64_t)D);
                    rms_fwd(xl, gl, eps, D, yl);
                    rms_fwd(xg, gg, eps, D, yg);
                    for (int d = 0; d < D; ++d) acc += (double)g[d] * (yg[d] - yl[d]);
                }
            }
            dp[bt] = z[bt] ? acc : 0.0;
        }
        free(yl);
        free(yg);
        free(dy);
    }
}

/* Gradients of the ContextNorm gains (Eq. 9, o~ = o * r * gain per head and
 * dimension) with z fixed as in oracle_combine_bwd.  o~ is linear in the gain,
 * so with dy the gradient reaching o~ (dy^L = dO (1 - p z), dy^G = dO p):
 *   dgL[h,d] = sum over every token of dy^L_d * oL_d * r^L
 *   dgG[h,d] = sum over the selected tokens of dy^G_d * oG_d * r^G
 * Summed in double over the tokens in order (b, t), serially. */
void oracle_combine_dgain(const float* dO, const float* oL, const float* oGc, const float* p,
                          const uint8_t* z, const int32_t* row_of, double eps, int B, int T, int H, int D,
                          double* dgL, double* dgG)
{
    int64_t ntok = (int64_t)B * T;
    memset(dgL, 0, sizeof(double) * (size_t)H * (size_t)D);
    memset(dgG, 0, sizeof(double) * (size_t)H * (size_t)D);
    for (int64_t bt = 0; bt < ntok; ++bt) {
        double pt = (double)p[bt];
        double wl = z[bt] ? 1.0 - pt : 1.0;
        for (int h = 0; h < H; ++h) {
            const float* g = dO + (bt * H + h) * (int64_t)D;
            const float* xl = oL + (bt * H + h) * (int64_t)D;
            double ss = 0.0;
            for (int d = 0; d < D; ++d) ss += (double)xl[d] * (double)xl[d];
            double rl = 1.0 / sqrt(ss / D + eps);
            for (int d = 0; d < D; ++d) dgL[(int64_t)h * D + d] += (double)g[d] * wl * (double)xl[d] * rl;
            if (z[bt]) {
                const float* xg = oGc + ((int64_t)row_of[bt] * H + h) * (int64_t)D;
                double sg = 0.0;
                for (int d = 0; d < D; ++d) sg += (double)xg[d] * (double)xg[d];
                double rg = 1.0 / sqrt(sg / D + eps);
                for (int d = 0; d < D; ++d) dgG[(int64_t)h * D + d] += (double)g[d] * pt * (double)xg[d] * rg;
            }
        }
    }
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
