/*
 * Float64 CPU oracle for the per-head spectral norm sigma_h = ||W^Q_h W^K_{g(h)}^T||_2.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the library path links or calls this file;
 * only tests/, the smoke check and the benchmark's CPU-baseline leg use it.  It
 * shares no code, header or constant with the CUDA library.
 *
 * Notation (paper, Section 3.1 and Appendix E): for one attention head,
 *   W^Q_h, W^K_g in R^{d x d_h},  M = W^Q_h W^K_g^T in R^{d x d}  (Eq. 4, bilinear form).
 * Weights arrive in the nn.Linear layout: the d_h x d row-major 16-bit block
 *   A[i][c] = W^Q_h[c][i]   (rows h*d_h .. h*d_h+d_h-1 of Wq),
 *   B[i][c] = W^K_g[c][i]   (rows g*d_h .. of Wk),
 * as bf16 (the default) or IEEE binary16 (oracle_set_weight_format(1)).  Every weight
 * is widened exactly to double; all arithmetic is double.
 *
 * Power iteration, Algorithm 2 (Appendix E.1), one "iteration" =
 *   u' = M v;  sigma = ||u'||;  u = u'/sigma;  v' = M^T u;  v = v'/||v'||.
 * The returned sigma is the one of the last iteration (||M v_{k-1}||).
 * Zero guard (the paper is silent): a zero start vector, or sigma == 0 at any
 * iteration, gives sigma = 0 and v_out = 0.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* 0: bf16 (the top 16 bits of an IEEE binary32); 1: IEEE binary16. */
static int g_weight_format = 0;

void oracle_set_weight_format(int fmt) { g_weight_format = fmt; }

/* binary16 by its definition: 1 sign bit, 5 exponent bits (bias 15), 10 fraction bits;
 * exponent 0 holds the subnormals f * 2^-24, exponent 31 infinities and NaNs. */
static double f16_bits_to_double(uint16_t bits)
{
    const int sign = (bits >> 15) & 1;
    const int e = (bits >> 10) & 0x1F;
    const int f = bits & 0x3FF;
    double mag;
    if (e == 0) mag = ldexp((double)f, -24);
    else if (e == 31) mag = f ? NAN : INFINITY;
    else mag = ldexp(1024.0 + f, e - 25);
    return sign ? -mag : mag;
}

static double bf16_to_double(uint16_t bits)
{
    if (g_weight_format == 1) return f16_bits_to_double(bits);
    union { uint32_t u; float f; } x;
    x.u = ((uint32_t)bits) << 16;
    return (double)x.f;
}

/* Decode n weights of the current format (for tests of the decoder). */
void oracle_decode_weights(const uint16_t *bits, long n, double *out)
{
    for (long i = 0; i < n; ++i) out[i] = bf16_to_double(bits[i]);
}

static double euclid_norm(const double *x, long n)
{
    double s = 0.0;
    for (long i = 0; i < n; ++i) s += x[i] * x[i];
    return sqrt(s);
}

/* M[r][c] = sum_i W^Q_h[r][i] W^K_g[c][i] = sum_i A[i][r] B[i][c]  (d x d, row-major). */
void oracle_form_interaction(int d, int dh, const uint16_t *A, const uint16_t *B, double *M)
{
    double *a = (double *)malloc(sizeof(double) * (size_t)dh);
    double *brow = (double *)malloc(sizeof(double) * (size_t)d);
    for (long r = 0; r < d; ++r) {
        double *mr = M + r * (long)d;
        for (long c = 0; c < d; ++c) mr[c] = 0.0;
        for (long i = 0; i < dh; ++i) a[i] = bf16_to_double(A[i * (long)d + r]);
        for (long i = 0; i < dh; ++i) {
            const uint16_t *bi = B + i * (long)d;
            for (long c = 0; c < d; ++c) brow[c] = bf16_to_double(bi[c]);
            for (long c = 0; c < d; ++c) mr[c] += a[i] * brow[c];
        }
    }
    free(a);
    free(brow);
}

/* Algorithm 2 on an explicitly formed d x d matrix M.  Returns 0 on success. */
int oracle_power_iteration_dense(int d, const double *M, const double *v0, int iters,
                                 double *sigma_out, double *v_out)
{
    double *v = (double *)malloc(sizeof(double) * (size_t)d);
    double *u = (double *)malloc(sizeof(double) * (size_t)d);
    double sigma = 0.0;
    int zero = 0;
    double nv = euclid_norm(v0, d);
    if (nv == 0.0) zero = 1;
    for (long c = 0; c < d && !zero; ++c) v[c] = v0[c] / nv;
    for (int t = 0; t < iters && !zero; ++t) {
        /* u' = M v */
        for (long r = 0; r < d; ++r) {
            double s = 0.0;
            const double *mr = M + r * (long)d;
            for (long c = 0; c < d; ++c) s += mr[c] * v[c];
            u[r] = s;
        }
        sigma = euclid_norm(u, d);
        if (sigma == 0.0) { zero = 1; break; }
        for (long r = 0; r < d; ++r) u[r] /= sigma;            /* u = u'/sigma */
        /* v' = M^T u */
        for (long c = 0; c < d; ++c) v[c] = 0.0;
        for (long r = 0; r < d; ++r) {
            const double *mr = M + r * (long)d;
            for (long c = 0; c < d; ++c) v[c] += mr[c] * u[r];
        }
        double nvp = euclid_norm(v, d);
        for (long c = 0; c < d; ++c) v[c] /= nvp;              /* v = v'/||v'|| */
    }
    if (zero) {
        sigma = 0.0;
        for (long c = 0; c < d; ++c) v[c] = 0.0;
    }
    *sigma_out = sigma;
    if (v_out) memcpy(v_out, v, sizeof(double) * (size_t)d);
    free(v);
    free(u);
    return 0;
}

/*
 * Algorithm 2 for one head with M applied in factored form (Section 4.1, Eqs. 18-19):
 *   z = W^K^T v  (z[i] = sum_c B[i][c] v[c]);     u' = W^Q z  (u'[c] = sum_i A[i][c] z[i]);
 *   y = W^Q^T u  (y[i] = sum_c A[i][c] u[c]);     v' = W^K y  (v'[c] = sum_i B[i][c] y[i]).
 */
int oracle_power_iteration_factored(int d, int dh, const uint16_t *A, const uint16_t *B,
                                    const double *v0, int iters, double *sigma_out, double *v_out)
{
    size_t nmat = (size_t)dh * (size_t)d;
    double *a = (double *)malloc(sizeof(double) * nmat);
    double *b = (double *)malloc(sizeof(double) * nmat);
    double *v = (double *)malloc(sizeof(double) * (size_t)d);
    double *u = (double *)malloc(sizeof(double) * (size_t)d);
    double *z = (double *)malloc(sizeof(double) * (size_t)dh);
    double *y = (double *)malloc(sizeof(double) * (size_t)dh);
    for (size_t e = 0; e < nmat; ++e) { a[e] = bf16_to_double(A[e]); b[e] = bf16_to_double(B[e]); }
    double sigma = 0.0;
    int zero = 0;
    double nv = euclid_norm(v0, d);
    if (nv == 0.0) zero = 1;
    for (long c = 0; c < d && !zero; ++c) v[c] = v0[c] / nv;
    for (int t = 0; t < iters && !zero; ++t) {
        for (long i = 0; i < dh; ++i) {                         /* z = W^K^T v */
            double s = 0.0;
            for (long c = 0; c < d; ++c) s += b[i * (long)d + c] * v[c];
            z[i] = s;
        }
        for (long c = 0; c < d; ++c) u[c] = 0.0;                /* u' = W^Q z */
        for (long i = 0; i < dh; ++i)
            for (long c = 0; c < d; ++c) u[c] += a[i * (long)d + c] * z[i];
        sigma = euclid_norm(u, d);                              /* sigma = ||u'|| */
        if (sigma == 0.0) { zero = 1; break; }
        for (long c = 0; c < d; ++c) u[c] /= sigma;             /* u = u'/sigma */
        for (long i = 0; i < dh; ++i) {                         /* y = W^Q^T u */
            double s = 0.0;
            for (long c = 0; c < d; ++c) s += a[i * (long)d + c] * u[c];
            y[i] = s;
        }
        for (long c = 0; c < d; ++c) v[c] = 0.0;                /* v' = W^K y */
        for (long i = 0; i < dh; ++i)
            for (long c = 0; c < d; ++c) v[c] += b[i * (long)d + c] * y[i];
        double nvp = euclid_norm(v, d);
        for (long c = 0; c < d; ++c) v[c] /= nvp;               /* v = v'/||v'|| */
    }
    if (zero) {
        sigma = 0.0;
        for (long c = 0; c < d; ++c) v[c] = 0.0;
    }
    *sigma_out = sigma;
    if (v_out) memcpy(v_out, v, sizeof(double) * (size_t)d);
    free(a); free(b); free(v); free(u); free(z); free(y);
    return 0;
}

/*
 * Per-head driver over a list of (layer, head) pairs.  wq[l] / wk[l] point at the
 * layer's bf16 Wq [n_q*d_h, d] / Wk [n_kv*d_h, d]; head h uses KV group
 * g(h) = h / (n_q/n_kv) (RepeatBlocks order, Appendix F).  v_in is float32
 * [layers][n_q][d]; outputs are indexed by position in the list.
 * mode 0: factored (Section 4.1);  mode 1: explicit M (d x d).
 */
int oracle_heads(int d, int n_q, int n_kv, int dh, const uint16_t *const *wq,
                 const uint16_t *const *wk, const float *v_in, int iters, int mode,
                 int count, const int *layer_idx, const int *head_idx,
                 double *sigma_out, double *v_out, int nthreads)
{
    if (n_kv <= 0 || n_q % n_kv != 0) return 1;
    int G = n_q / n_kv;
    int rc = 0;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#pragma omp parallel for schedule(dynamic, 1)
#endif
    for (int j = 0; j < count; ++j) {
        int l = layer_idx[j], h = head_idx[j];
        int g = h / G;
        const uint16_t *A = wq[l] + (size_t)h * dh * d;
        const uint16_t *B = wk[l] + (size_t)g * dh * d;
        double *v0 = (double *)malloc(sizeof(double) * (size_t)d);
        const float *vf = v_in + ((size_t)l * n_q + h) * (size_t)d;
        for (long c = 0; c < d; ++c) v0[c] = (double)vf[c];
        double *vo = v_out ? v_out + (size_t)j * d : NULL;
        if (mode == 1) {
            double *M = (double *)malloc(sizeof(double) * (size_t)d * (size_t)d);
            if (!M) { rc = 2; free(v0); continue; }
            oracle_form_interaction(d, dh, A, B, M);
            oracle_power_iteration_dense(d, M, v0, iters, &sigma_out[j], vo);
            free(M);
        } else {
            oracle_power_iteration_factored(d, dh, A, B, v0, iters, &sigma_out[j], vo);
        }
        free(v0);
    }
    return rc;
}

/*
 * Whole-layer form, exactly Algorithm 3 (Appendix E.2): W^Q in R^{d x n_q d_h},
 * W^K in R^{d x n_kv d_h}, M = W^Q W^K_exp^T with W^K_exp repeating each d_h
 * block of W^K g times (Section 4.2).
 *   z_kv = W^K^T v;  z = RepeatBlocks(z_kv, g);  u' = W^Q z;  sigma = ||u'||; u = u'/sigma;
 *   y = W^Q^T u;  y_kv = SumGroups(y, g);  v' = W^K y_kv;  v = v'/||v'||.
 * Wq / Wk are the layer's nn.Linear blocks ([n_q*d_h, d], [n_kv*d_h, d]).
 */
int oracle_layer_implicit_gqa(int d, int n_q, int n_kv, int dh, const uint16_t *Wq,
                              const uint16_t *Wk, const double *v0, int iters,
                              double *sigma_out, double *v_out)
{
    if (n_kv <= 0 || n_q % n_kv != 0) return 1;
    int g = n_q / n_kv;
    long rq = (long)n_q * dh, rk = (long)n_kv * dh;
    double *v = (double *)malloc(sizeof(double) * (size_t)d);
    double *u = (double *)malloc(sizeof(double) * (size_t)d);
    double *zkv = (double *)malloc(sizeof(double) * (size_t)rk);
    double *z = (double *)malloc(sizeof(double) * (size_t)rq);
    double *y = (double *)malloc(sizeof(double) * (size_t)rq);
    double *ykv = (double *)malloc(sizeof(double) * (size_t)rk);
    double sigma = 0.0;
    int zero = 0;
    double nv = euclid_norm(v0, d);
    if (nv == 0.0) zero = 1;
    for (long c = 0; c < d && !zero; ++c) v[c] = v0[c] / nv;
    for (int t = 0; t < iters && !zero; ++t) {
        for (long r = 0; r < rk; ++r) {                         /* z_kv = W^K^T v */
            double s = 0.0;
            for (long c = 0; c < d; ++c) s += bf16_to_double(Wk[r * d + c]) * v[c];
            zkv[r] = s;
        }
        for (long hq = 0; hq < n_q; ++hq)                       /* RepeatBlocks(z_kv, g) */
            for (long i = 0; i < dh; ++i) z[hq * dh + i] = zkv[(hq / g) * dh + i];
        for (long c = 0; c < d; ++c) u[c] = 0.0;                /* u' = W^Q z */
        for (long r = 0; r < rq; ++r)
            for (long c = 0; c < d; ++c) u[c] += bf16_to_double(Wq[r * d + c]) * z[r];
        sigma = euclid_norm(u, d);
        if (sigma == 0.0) { zero = 1; break; }
        for (long c = 0; c < d; ++c) u[c] /= sigma;
        for (long r = 0; r < rq; ++r) {                         /* y = W^Q^T u */
            double s = 0.0;
            for (long c = 0; c < d; ++c) s += bf16_to_double(Wq[r * d + c]) * u[c];
            y[r] = s;
        }
        for (long r = 0; r < rk; ++r) ykv[r] = 0.0;             /* SumGroups(y, g) */
        for (long hq = 0; hq < n_q; ++hq)
            for (long i = 0; i < dh; ++i) ykv[(hq / g) * dh + i] += y[hq * dh + i];
        for (long c = 0; c < d; ++c) v[c] = 0.0;                /* v' = W^K y_kv */
        for (long r = 0; r < rk; ++r)
            for (long c = 0; c < d; ++c) v[c] += bf16_to_double(Wk[r * d + c]) * ykv[r];
        double nvp = euclid_norm(v, d);
        for (long c = 0; c < d; ++c) v[c] /= nvp;
    }
    if (zero) {
        sigma = 0.0;
        for (long c = 0; c < d; ++c) v[c] = 0.0;
    }
    *sigma_out = sigma;
    if (v_out) memcpy(v_out, v, sizeof(double) * (size_t)d);
    free(v); free(u); free(zkv); free(z); free(y); free(ykv);
    return 0;
}

/*
 * The explicit expansion that Section 4.2 avoids: W^K_exp in R^{d x n_q d_h}
 * (row block hq*d_h.. of the nn.Linear layout copies block (hq/g)*d_h.. of Wk),
 * then M = W^Q W^K_exp^T formed densely.  Writes M (d x d).
 */
int oracle_layer_form_expanded(int d, int n_q, int n_kv, int dh, const uint16_t *Wq,
                               const uint16_t *Wk, double *M)
{
    if (n_kv <= 0 || n_q % n_kv != 0) return 1;
    int g = n_q / n_kv;
    long rq = (long)n_q * dh;
    uint16_t *wkexp = (uint16_t *)malloc(sizeof(uint16_t) * (size_t)rq * (size_t)d);
    for (long hq = 0; hq < n_q; ++hq)
        for (long i = 0; i < dh; ++i)
            memcpy(wkexp + (hq * dh + i) * (long)d, Wk + ((hq / g) * dh + i) * (long)d,
                   sizeof(uint16_t) * (size_t)d);
    /* M[r][c] = sum_j W^Q[r][j] W^K_exp[c][j], j over all n_q*d_h columns */
    oracle_form_interaction(d, (int)rq, Wq, wkexp, M);
    free(wkexp);
    return 0;
}

#ifdef _OPENMP
int oracle_max_threads(void) { return omp_get_max_threads(); }
#else
int oracle_max_threads(void) { return 1; }
#endif
