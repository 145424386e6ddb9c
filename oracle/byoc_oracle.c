/*
 * byoc_oracle.c -- fp64 CPU oracle for the offloaded composite regions.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product library links, includes
 * or calls this file; only the tests, the smoke check and the CPU-baseline leg
 * of the benchmark load it.  It shares no code, header, table or helper with
 * the CUDA path.
 *
 * Every routine is a plain direct loop over the textbook definition of one
 * operator of the paper's composite patterns (Section 3.1.1, the
 * Conv2D-Add-ReLU listing; Section 3.1 names the operator attributes stride,
 * padding and dilation).  All arithmetic is double precision; the summation
 * order is the natural loop order.  Layout is NHWC for activations
 * (Section 3.2, layout transformation), OIHW for convolution weights and
 * [units, in] for dense weights.  There is no blocking, fusion or reordering.
 *
 * Operator definitions (the paper gives none; these are the standard
 * inference-time definitions):
 *   conv2d       y[n,p,q,k] = sum_{c in group(k), r, s}
 *                  x[n, p*sh + r*dh - pt, q*sw + s*dw - pl, c] * w[k, c', r, s]
 *                (cross-correlation; x is zero outside the image)
 *   dense        y[m,u] = sum_i x[m,i] * w[u,i]
 *   bias_add     y[...,c] += b[c]
 *   batch_norm   y = gamma*(x-mean)/sqrt(var+eps) + beta   (inference form)
 *   relu         max(x,0)          relu6  min(max(x,0),6)
 *   gelu         0.5*x*(1+erf(x/sqrt(2)))                   (erf form)
 *   add          y = a + b (same shape)
 *   max_pool2d   max over the window, padding never selected
 *   global_avg   mean over H and W
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>

#define OIDX4(a, b, c, d, B, C, D) ((((size_t)(a) * (B) + (b)) * (C) + (c)) * (D) + (d))

/* conv2d, NHWC input [N,H,W,C], OIHW weight [K, C/groups, R, S],
 * NHWC output [N,Ho,Wo,K].  pad = {top, left, bottom, right}. */
void oracle_conv2d_nhwc(const double *x, int N, int H, int W, int C,
                        const double *w, int K, int R, int S, int groups,
                        int sh, int sw, int pt, int pl, int pb, int pr,
                        int dh, int dw, double *y) {
    int Ho = (H + pt + pb - dh * (R - 1) - 1) / sh + 1;
    int Wo = (W + pl + pr - dw * (S - 1) - 1) / sw + 1;
    int Cg = C / groups;      /* input channels per group */
    int Kg = K / groups;      /* output channels per group */
    long total = (long)N * Ho * Wo;
#pragma omp parallel for schedule(static)
    for (long pix = 0; pix < total; ++pix) {
        int n = (int)(pix / ((long)Ho * Wo));
        int rem = (int)(pix % ((long)Ho * Wo));
        int p = rem / Wo, q = rem % Wo;
        for (int k = 0; k < K; ++k) {
            int g = k / Kg;
            double acc = 0.0;
            for (int ci = 0; ci < Cg; ++ci) {
                int c = g * Cg + ci;
                for (int r = 0; r < R; ++r) {
                    int h = p * sh + r * dh - pt;
                    if (h < 0 || h >= H) continue;
                    for (int s = 0; s < S; ++s) {
                        int ww = q * sw + s * dw - pl;
                        if (ww < 0 || ww >= W) continue;
                        acc += x[OIDX4(n, h, ww, c, H, W, C)] *
                               w[OIDX4(k, ci, r, s, Cg, R, S)];
                    }
                }
            }
            y[(size_t)pix * K + k] = acc;
        }
    }
}

/* The same conv2d evaluated only at `count` chosen outputs: output pixel
 * index pix[i] (flattened n,p,q) and output channel ks[i]. */
void oracle_conv2d_nhwc_sampled(const double *x, int N, int H, int W, int C,
                                const double *w, int K, int R, int S, int groups,
                                int sh, int sw, int pt, int pl, int pb, int pr,
                                int dh, int dw, const long *pix, const int *ks,
                                long count, double *out) {
    int Ho = (H + pt + pb - dh * (R - 1) - 1) / sh + 1;
    int Wo = (W + pl + pr - dw * (S - 1) - 1) / sw + 1;
    int Cg = C / groups, Kg = K / groups;
    (void)N;
#pragma omp parallel for schedule(static)
    for (long i = 0; i < count; ++i) {
        int n = (int)(pix[i] / ((long)Ho * Wo));
        int rem = (int)(pix[i] % ((long)Ho * Wo));
        int p = rem / Wo, q = rem % Wo, k = ks[i], g = k / Kg;
        double acc = 0.0;
        for (int ci = 0; ci < Cg; ++ci) {
            int c = g * Cg + ci;
            for (int r = 0; r < R; ++r) {
                int h = p * sh + r * dh - pt;
                if (h < 0 || h >= H) continue;
                for (int s = 0; s < S; ++s) {
                    int ww = q * sw + s * dw - pl;
                    if (ww < 0 || ww >= W) continue;
                    acc += x[OIDX4(n, h, ww, c, H, W, C)] * w[OIDX4(k, ci, r, s, Cg, R, S)];
                }
            }
        }
        out[i] = acc;
    }
}

/* dense: x [M, I] row-major, w [U, I] (units x in), y [M, U]. */
void oracle_dense(const double *x, int M, int I, const double *w, int U,
                  double *y) {
#pragma omp parallel for schedule(static)
    for (int m = 0; m < M; ++m) {
        for (int u = 0; u < U; ++u) {
            double acc = 0.0;
            for (int i = 0; i < I; ++i)
                acc += x[(size_t)m * I + i] * w[(size_t)u * I + i];
            y[(size_t)m * U + u] = acc;
        }
    }
}

/* bias_add on the innermost (channel) axis, in place; rows = elements / C. */
void oracle_bias_add(double *y, long rows, int C, const double *b) {
#pragma omp parallel for schedule(static)
    for (long i = 0; i < rows; ++i)
        for (int c = 0; c < C; ++c) y[i * C + c] += b[c];
}

/* batch_norm in inference form on the channel axis, in place. */
void oracle_batch_norm(double *y, long rows, int C, const double *gamma,
                       const double *beta, const double *mean,
                       const double *var, double eps) {
#pragma omp parallel for schedule(static)
    for (long i = 0; i < rows; ++i)
        for (int c = 0; c < C; ++c) {
            double v = y[i * C + c];
            y[i * C + c] = gamma[c] * (v - mean[c]) / sqrt(var[c] + eps) + beta[c];
        }
}

void oracle_relu(double *y, long n) {
#pragma omp parallel for schedule(static)
    for (long i = 0; i < n; ++i) y[i] = y[i] > 0.0 ? y[i] : 0.0;
}

void oracle_relu6(double *y, long n) {
#pragma omp parallel for schedule(static)
    for (long i = 0; i < n; ++i) {
        double v = y[i] > 0.0 ? y[i] : 0.0;
        y[i] = v < 6.0 ? v : 6.0;
    }
}

void oracle_gelu(double *y, long n) {
    const double inv_sqrt2 = 0.70710678118654752440;
#pragma omp parallel for schedule(static)
    for (long i = 0; i < n; ++i) y[i] = 0.5 * y[i] * (1.0 + erf(y[i] * inv_sqrt2));
}

/* y += a, elementwise. */
void oracle_add(double *y, const double *a, long n) {
#pragma omp parallel for schedule(static)
    for (long i = 0; i < n; ++i) y[i] += a[i];
}

/* max_pool2d, NHWC; positions outside the image never win. */
void oracle_max_pool2d_nhwc(const double *x, int N, int H, int W, int C,
                            int R, int S, int sh, int sw, int pt, int pl,
                            int pb, int pr, double *y) {
    int Ho = (H + pt + pb - R) / sh + 1;
    int Wo = (W + pl + pr - S) / sw + 1;
    long total = (long)N * Ho * Wo;
#pragma omp parallel for schedule(static)
    for (long pix = 0; pix < total; ++pix) {
        int n = (int)(pix / ((long)Ho * Wo));
        int rem = (int)(pix % ((long)Ho * Wo));
        int p = rem / Wo, q = rem % Wo;
        for (int c = 0; c < C; ++c) {
            double best = -INFINITY;
            for (int r = 0; r < R; ++r) {
                int h = p * sh + r - pt;
                if (h < 0 || h >= H) continue;
                for (int s = 0; s < S; ++s) {
                    int ww = q * sw + s - pl;
                    if (ww < 0 || ww >= W) continue;
                    double v = x[OIDX4(n, h, ww, c, H, W, C)];
                    if (v > best) best = v;
                }
            }
            y[(size_t)pix * C + c] = best;
        }
    }
}

/* global average pool, NHWC [N,H,W,C] -> [N,C]. */
void oracle_global_avg_pool_nhwc(const double *x, int N, int H, int W, int C,
                                 double *y) {
#pragma omp parallel for schedule(static)
    for (int n = 0; n < N; ++n)
        for (int c = 0; c < C; ++c) {
            double acc = 0.0;
            for (int h = 0; h < H; ++h)
                for (int ww = 0; ww < W; ++ww) acc += x[OIDX4(n, h, ww, c, H, W, C)];
            y[(size_t)n * C + c] = acc / ((double)H * W);
        }
}

/* Number of OpenMP threads the oracle runs with (1 when built without it). */
int oracle_num_threads(void) {
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_num_threads(int n) {
#ifdef _OPENMP
    extern void omp_set_num_threads(int);
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}
