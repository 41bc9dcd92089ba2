/*
 * Plain fp64 CPU oracle for scaled dot-product attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call this code:
 * it exists so that the tests, the self-check in __graft_entry__.smoke() and
 * the timed CPU baseline of bench.py have an obviously correct answer to
 * compare the CUDA kernels against.  It shares no code, header, table or helper
 * with the CUDA library.
 *
 * What it computes (paper Section 4, Eq. attention with the stable softmax of
 * Eq. stable_softmax, and the output contraction of Eq. output_dnf):
 *
 *     O[b,h,i,c] = sum_k w[b,h,i,k] * V[b,h,k,c]
 *     w[b,h,i,k] = exp(s[k] - m) / sum_k' exp(s[k'] - m)
 *     s[k]       = scale * sum_j Q[b,h,i,j] * K[b,h,k,j],   m = max_k s[k]
 *
 * Each (b,h) slice is an independent 2-D problem (Remark in Section 4.2), and
 * within a slice every output row is computed on its own, in the order of the
 * paper's Algorithm 1 (Section 7.1): scores for all keys, row maximum,
 * exponentials, their sum, the normalised weights, then the weighted sum of the
 * value rows.  The scratch vectors s, e, w are O(N_k) per row, as the paper
 * notes after Algorithm 1.
 *
 * Arithmetic is IEEE double with libm exp(); every reduction runs in index
 * order, sequentially.  Compile without -ffast-math and with
 * -ffp-contract=off so that no multiply-add is fused: results are then the
 * same on x86-64 and AArch64.  OpenMP splits the work over whole rows only, so
 * the result is bit-identical for any thread count.
 *
 * moa_oracle_attn_lse_f64 also returns each row's log-sum-exp, moa_oracle_attn_bwd_f64 the
 * gradients dQ, dK, dV of the backward pass (Stage 5, Section 9) for a given dL/dO, and
 * moa_oracle_qkv_proj_f64 the input projections Q = X W_Q, K = X W_K, V = X W_V (Section 4.1).
 *
 * Inputs are float32 arrays holding the stored values exactly (bf16 and fp32
 * values both embed exactly in float32); every element is widened to double
 * before use.  scale is taken as given (the paper fixes 1/sqrt(d_k)).
 *
 * Return value of every entry point: 0 on success, -1 on a bad argument,
 * -2 if scratch memory could not be allocated.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    const float *Q, *K, *V;
    int64_t B, H, Nq, Nk, dk, dv;
    double scale;
} oracle_problem;

static int check_problem(const oracle_problem *p)
{
    if (!p->Q || !p->K || !p->V) return -1;
    if (p->B <= 0 || p->H <= 0 || p->Nq <= 0 || p->Nk <= 0 || p->dk <= 0 || p->dv <= 0) return -1;
    return 0;
}

/* Step 1 of Algorithm 1 for one row: the scaled scores s[k] (Eq. mm_psi reads
 * K by row k, so no transposed copy of K is formed). */
static void row_scores(const oracle_problem *p, int64_t row, double *s)
{
    const int64_t bh = row / p->Nq;
    const int64_t i = row % p->Nq;
    const float *q = p->Q + (bh * p->Nq + i) * p->dk;
    const float *Kh = p->K + bh * p->Nk * p->dk;
    for (int64_t k = 0; k < p->Nk; ++k) {
        const float *kr = Kh + k * p->dk;
        double dot = 0.0;
        for (int64_t j = 0; j < p->dk; ++j)
            dot += (double)q[j] * (double)kr[j];
        s[k] = dot * p->scale;
    }
}

/* Steps 2-5 of Algorithm 1 for one row, given its scores: row maximum (Step I
 * of Section 4.3), exponentials of the shifted scores (Step II), their sum
 * (Step III), division (Step IV), then the contraction with V (Eq.
 * output_dnf).  w_out, if not NULL, receives the weights; o_out, if not NULL,
 * receives the output row. */
static void row_softmax_output(const oracle_problem *p, int64_t row, double *s, double *e,
                               double *w, double *w_out, double *o_out, double *lse_out)
{
    const int64_t bh = row / p->Nq;
    const float *Vh = p->V + bh * p->Nk * p->dv;
    double m = s[0];
    for (int64_t k = 1; k < p->Nk; ++k)
        if (s[k] > m) m = s[k];
    for (int64_t k = 0; k < p->Nk; ++k)
        e[k] = exp(s[k] - m);
    double Z = 0.0;
    for (int64_t k = 0; k < p->Nk; ++k)
        Z += e[k];
    for (int64_t k = 0; k < p->Nk; ++k)
        w[k] = e[k] / Z;
    /* log of the denominator of Eq. stable_softmax before the shift: ln sum_k exp(s[k]) */
    if (lse_out) *lse_out = m + log(Z);
    if (w_out)
        for (int64_t k = 0; k < p->Nk; ++k)
            w_out[k] = w[k];
    if (o_out)
        for (int64_t c = 0; c < p->dv; ++c) {
            double acc = 0.0;
            for (int64_t k = 0; k < p->Nk; ++k)
                acc += w[k] * (double)Vh[k * p->dv + c];
            o_out[c] = acc;
        }
}

/* Common driver: rows[r] (or r itself when rows == NULL) for r < nrows.
 * shift, if not NULL, adds shift[r] to every score of output row r before the
 * softmax (used only to test shift invariance). */
static int run_rows(const oracle_problem *p, const int64_t *rows, int64_t nrows,
                    const double *shift, double *W, double *S, double *O, double *LSE,
                    int nthreads)
{
    if (check_problem(p)) return -1;
    if (nrows < 0) return -1;
    const int64_t total = p->B * p->H * p->Nq;
    if (rows)
        for (int64_t r = 0; r < nrows; ++r)
            if (rows[r] < 0 || rows[r] >= total) return -1;
    int status = 0;
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel num_threads(nthreads)
#endif
    {
        double *buf = (double *)malloc(sizeof(double) * 3 * (size_t)p->Nk);
        if (!buf) {
#ifdef _OPENMP
#pragma omp atomic write
#endif
            status = -2;
        } else {
            double *s = buf, *e = buf + p->Nk, *w = buf + 2 * p->Nk;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
            for (int64_t r = 0; r < nrows; ++r) {
                const int64_t row = rows ? rows[r] : r;
                row_scores(p, row, s);
                if (shift)
                    for (int64_t k = 0; k < p->Nk; ++k)
                        s[k] = s[k] + shift[r];
                if (S)
                    for (int64_t k = 0; k < p->Nk; ++k)
                        S[r * p->Nk + k] = s[k];
                row_softmax_output(p, row, s, e, w, W ? W + r * p->Nk : NULL,
                                   O ? O + r * p->dv : NULL, LSE ? LSE + r : NULL);
            }
            free(buf);
        }
    }
    return status;
}

/* O[B,H,Nq,dv] for the whole problem. */
int moa_oracle_attn_f64(const float *Q, const float *K, const float *V, double *O, int64_t B,
                        int64_t H, int64_t Nq, int64_t Nk, int64_t dk, int64_t dv, double scale,
                        int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!O) return -1;
    return run_rows(&p, NULL, check_problem(&p) ? 0 : B * H * Nq, NULL, NULL, NULL, O, NULL, nthreads);
}

/* Output rows for a list of flattened row indices r = (b*H + h)*Nq + i;
 * O receives nrows x dv values. */
int moa_oracle_rows_f64(const float *Q, const float *K, const float *V, double *O, int64_t B,
                        int64_t H, int64_t Nq, int64_t Nk, int64_t dk, int64_t dv, double scale,
                        const int64_t *rows, int64_t nrows, int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!O || !rows) return -1;
    return run_rows(&p, rows, nrows, NULL, NULL, NULL, O, NULL, nthreads);
}

/* Attention weights W[B,H,Nq,Nk] (Eq. dnf_attn) and, if O is not NULL, the
 * output as well.  Meant for small problems. */
int moa_oracle_weights_f64(const float *Q, const float *K, const float *V, double *W, double *O,
                           int64_t B, int64_t H, int64_t Nq, int64_t Nk, int64_t dk, int64_t dv,
                           double scale, int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!W) return -1;
    return run_rows(&p, NULL, check_problem(&p) ? 0 : B * H * Nq, NULL, W, NULL, O, NULL, nthreads);
}

/* Scaled scores S[B,H,Nq,Nk] (Step 1 of Algorithm 1 only).  Meant for small
 * problems and for checking properties of generated inputs. */
int moa_oracle_scores_f64(const float *Q, const float *K, int64_t B, int64_t H, int64_t Nq,
                          int64_t Nk, int64_t dk, double scale, double *S, int nthreads)
{
    oracle_problem p = {Q, K, K, B, H, Nq, Nk, dk, 1, scale};
    if (!S || check_problem(&p)) return -1;
    const int64_t total = B * H * Nq;
    int status = 0;
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 16) num_threads(nthreads)
#endif
    for (int64_t r = 0; r < total; ++r)
        row_scores(&p, r, S + r * Nk);
    return status;
}

/* Same as moa_oracle_attn_f64 but adds shift[r] to every score of row r
 * before the softmax.  By Eq. stable_softmax the result must not depend on
 * shift; the tests use this to check that property. */
int moa_oracle_attn_shifted_f64(const float *Q, const float *K, const float *V, double *O,
                                int64_t B, int64_t H, int64_t Nq, int64_t Nk, int64_t dk,
                                int64_t dv, double scale, const double *shift, int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!O || !shift) return -1;
    return run_rows(&p, NULL, check_problem(&p) ? 0 : B * H * Nq, shift, NULL, NULL, O, NULL, nthreads);
}

/* Output O and, per output row, LSE = ln sum_k exp(s[k]) (the scaled scores' log-sum-exp,
 * i.e. m + ln Z of Algorithm 1); LSE has B*H*Nq entries. */
int moa_oracle_attn_lse_f64(const float *Q, const float *K, const float *V, double *O,
                            double *LSE, int64_t B, int64_t H, int64_t Nq, int64_t Nk,
                            int64_t dk, int64_t dv, double scale, int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!O || !LSE) return -1;
    return run_rows(&p, NULL, check_problem(&p) ? 0 : B * H * Nq, NULL, NULL, NULL, O, LSE,
                    nthreads);
}

/*
 * Backward pass of Eq. attention (paper Stage 5, Section 9).  With L a scalar loss and
 * dO = dL/dO given, the paper writes the query gradient as
 *     dL/dQ = dL/dO . V^T . (d softmax / d scaled scores) . K * scale,
 * where the softmax Jacobian of one row with weights w is J = diag(w) - w w^T (dense N_k x N_k).
 * J is symmetric and is applied here without being formed: for dP = dO V^T (one row),
 *     J dP = w * (dP - w.dP)      (elementwise; w.dP is one number per row).
 * dK and dV follow from the same chain rule applied to the other two operands of Eq.
 * attention (the paper derives only dQ; these are the standard derivatives of the same
 * expression):
 *     dS = J dP (per row),  dQ = scale * dS K,  dK = scale * dS^T Q,  dV = W^T dO.
 * One (b,h) slice per thread; inside a slice the rows are taken in index order, so the
 * dK and dV sums have a fixed order and the result does not depend on the thread count.
 * dQ is [B,H,Nq,dk], dK [B,H,Nk,dk], dV [B,H,Nk,dv].
 */
int moa_oracle_attn_bwd_f64(const float *Q, const float *K, const float *V, const float *dO,
                            double *dQ, double *dK, double *dV, int64_t B, int64_t H,
                            int64_t Nq, int64_t Nk, int64_t dk, int64_t dv, double scale,
                            int nthreads)
{
    oracle_problem p = {Q, K, V, B, H, Nq, Nk, dk, dv, scale};
    if (!dO || !dQ || !dK || !dV || check_problem(&p)) return -1;
    int status = 0;
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel num_threads(nthreads)
#endif
    {
        double *buf = (double *)malloc(sizeof(double) * 5 * (size_t)Nk);
        if (!buf) {
#ifdef _OPENMP
#pragma omp atomic write
#endif
            status = -2;
        } else {
            double *s = buf, *e = buf + Nk, *w = buf + 2 * Nk, *dP = buf + 3 * Nk;
            double *dS = buf + 4 * Nk;
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 1)
#endif
            for (int64_t bh = 0; bh < B * H; ++bh) {
                const float *Kh = K + bh * Nk * dk;
                const float *Vh = V + bh * Nk * dv;
                double *dKh = dK + bh * Nk * dk;
                double *dVh = dV + bh * Nk * dv;
                for (int64_t t = 0; t < Nk * dk; ++t) dKh[t] = 0.0;
                for (int64_t t = 0; t < Nk * dv; ++t) dVh[t] = 0.0;
                for (int64_t i = 0; i < Nq; ++i) {
                    const int64_t row = bh * Nq + i;
                    const float *q = Q + row * dk;
                    const float *g = dO + row * dv;
                    /* forward weights of this row (Algorithm 1) */
                    row_scores(&p, row, s);
                    row_softmax_output(&p, row, s, e, w, NULL, NULL, NULL);
                    /* dP = dO_i V^T, then the Jacobian product dS = w * (dP - w.dP) */
                    for (int64_t k = 0; k < Nk; ++k) {
                        double acc = 0.0;
                        for (int64_t c = 0; c < dv; ++c)
                            acc += (double)g[c] * (double)Vh[k * dv + c];
                        dP[k] = acc;
                    }
                    double wdp = 0.0;
                    for (int64_t k = 0; k < Nk; ++k)
                        wdp += w[k] * dP[k];
                    for (int64_t k = 0; k < Nk; ++k)
                        dS[k] = w[k] * (dP[k] - wdp);
                    /* dQ_i = scale * dS K */
                    for (int64_t j = 0; j < dk; ++j) {
                        double acc = 0.0;
                        for (int64_t k = 0; k < Nk; ++k)
                            acc += dS[k] * (double)Kh[k * dk + j];
                        dQ[row * dk + j] = scale * acc;
                    }
                    /* dK_k += scale * dS_k q_i,  dV_k += w_k dO_i */
                    for (int64_t k = 0; k < Nk; ++k) {
                        for (int64_t j = 0; j < dk; ++j)
                            dKh[k * dk + j] += scale * dS[k] * (double)q[j];
                        for (int64_t c = 0; c < dv; ++c)
                            dVh[k * dv + c] += w[k] * (double)g[c];
                    }
                }
            }
            free(buf);
        }
    }
    return status;
}

/*
 * Input projections of Section 4.1: Q = X W_Q, K = X W_K, V = X W_V, for X [B, N, d] and the
 * three weight matrices side by side in one row-major array W [d, H*dk + H*dk + H*dv]
 * (columns [0, H*dk) are W_Q, then W_K, then W_V).  Column h*dk + j of W_Q produces feature j
 * of head h, and the results are stored head-major, as the attention entry points take them:
 *     Q[b,h,n,j] = sum_c X[b,n,c] W[c, h*dk + j]
 *     K[b,h,n,j] = sum_c X[b,n,c] W[c, H*dk + h*dk + j]
 *     V[b,h,n,j] = sum_c X[b,n,c] W[c, 2*H*dk + h*dv + j]
 * Plain fp64 dot products in index order.
 */
int moa_oracle_qkv_proj_f64(const float *X, const float *W, double *Q, double *K, double *V,
                            int64_t B, int64_t N, int64_t d, int64_t H, int64_t dk, int64_t dv,
                            int nthreads)
{
    if (!X || !W || !Q || !K || !V) return -1;
    if (B <= 0 || N <= 0 || d <= 0 || H <= 0 || dk <= 0 || dv <= 0) return -1;
    const int64_t ncol = 2 * H * dk + H * dv;
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel for schedule(dynamic, 16) num_threads(nthreads)
#endif
    for (int64_t t = 0; t < B * N; ++t) {
        const int64_t b = t / N, n = t % N;
        const float *x = X + t * d;
        for (int64_t col = 0; col < ncol; ++col) {
            double acc = 0.0;
            for (int64_t c = 0; c < d; ++c)
                acc += (double)x[c] * (double)W[c * ncol + col];
            if (col < H * dk) {
                const int64_t h = col / dk, j = col % dk;
                Q[((b * H + h) * N + n) * dk + j] = acc;
            } else if (col < 2 * H * dk) {
                const int64_t h = (col - H * dk) / dk, j = (col - H * dk) % dk;
                K[((b * H + h) * N + n) * dk + j] = acc;
            } else {
                const int64_t h = (col - 2 * H * dk) / dv, j = (col - 2 * H * dk) % dv;
                V[((b * H + h) * N + n) * dv + j] = acc;
            }
        }
    }
    return 0;
}

/* Threads an OpenMP region would use by default (1 without OpenMP). */
int moa_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
