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

/* Threads an OpenMP region would use by default (1 without OpenMP). */
int moa_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
