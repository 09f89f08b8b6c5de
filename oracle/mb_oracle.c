/*
 * fp64 CPU oracle for the MambaByte selective-scan layer core.
 *
 * TEST INFRASTRUCTURE. This file is the plain, slow, sequential definition
 * that the CUDA kernels are checked against. Only the test suite, the smoke
 * check and the benchmark's CPU-baseline leg may load it; the library's
 * product path never calls it and shares no code with it.
 *
 * What it computes (MambaByte, Section 2 "Selective SSMs", Eq. 1-3, and
 * Appendix "Discretization and selection"):
 *
 *   for every batch row b and channel d (independent of each other):
 *     h[n] = h0[b,d,n]   (zeros when h0 is NULL)
 *     for t = 0 .. L-1:
 *       Delta   = softplus(dt[b,t,d] + dt_bias[d])            Eq. 3
 *       Abar[n] = exp(Delta * A[d,n])                          ZOH for A
 *       Bbar[n] = Delta * B[b,t,n]                              Euler for B
 *                 (or (exp(Delta*A)-1)/A * B with the ZOH rule)
 *       h[n]    = Abar[n] * h[n] + Bbar[n] * x[b,t,d]           Eq. 2
 *       y       = sum_n C[b,t,n] * h[n] + D[d] * x[b,t,d]       Table 6 "Output"
 *       out     = y * silu(z[b,t,d])   (no gate when z NULL)   Fig. 6, Table 6 "gating"
 *       h_all[b,t,d,n] = h[n]          (when h_all is given)   Algorithm 1, verify
 *     h_last[b,d,n] = h[n]
 *
 * Eq. 2 uses the updated state h[k] in y[k]; the recurrence is evaluated in
 * the order it is written, one time step after the other, in fp64.
 *
 * Layouts (all row-major, contiguous): x, z, dt, y [batch, L, D]; B, C
 * [batch, L, N]; A [D, N]; D, dt_bias [D]; h0, h_last [batch, D, N];
 * h_all [batch, L, D, N].
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* softplus(v) = log(1 + e^v), evaluated without overflow. */
static double softplus(double v) { return fmax(v, 0.0) + log1p(exp(-fabs(v))); }

/* silu(z) = z * sigmoid(z) (the Swish gate of the Mamba block). */
static double silu(double z) { return z / (1.0 + exp(-z)); }

/* B discretisation rules: 0 = Euler (Bbar = Delta*B, what Mamba uses, per the
 * footnote of the discretisation appendix), 1 = zero-order hold
 * (Bbar = A^-1 (exp(A Delta) - 1) B, the appendix formula; Delta*B when A = 0). */
enum { ORACLE_B_EULER = 0, ORACLE_B_ZOH = 1 };

int oracle_scan(int64_t batch, int64_t L, int64_t Dn, int64_t N,
                const double *x, const double *z, const double *dt,
                const double *B, const double *C, const double *A,
                const double *Dskip, const double *dt_bias, const double *h0,
                int b_rule, double *y, double *h_last, double *h_all,
                int nthreads)
{
    if (batch < 0 || L < 0 || Dn < 0 || N <= 0) return 1;
    if (nthreads < 1) nthreads = 1;
    int64_t nchan = batch * Dn;
    int err = 0;
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 4) reduction(| : err)
    for (int64_t ch = 0; ch < nchan; ++ch) {
        int64_t b = ch / Dn, d = ch % Dn;
        double *h = (double *)malloc((size_t)N * sizeof(double));
        if (!h) { err |= 1; continue; }
        for (int64_t n = 0; n < N; ++n)
            h[n] = h0 ? h0[(b * Dn + d) * N + n] : 0.0;
        for (int64_t t = 0; t < L; ++t) {
            int64_t i = (b * L + t) * Dn + d;       /* [b, t, d] */
            const double *Bt = B + (b * L + t) * N; /* [b, t, :] */
            const double *Ct = C + (b * L + t) * N;
            double delta = softplus(dt[i] + (dt_bias ? dt_bias[d] : 0.0));
            double acc = 0.0;
            for (int64_t n = 0; n < N; ++n) {
                double a = A[d * N + n];
                double abar = exp(delta * a);
                double bbar;
                if (b_rule == ORACLE_B_ZOH && a != 0.0)
                    bbar = (abar - 1.0) / a * Bt[n];
                else
                    bbar = delta * Bt[n];
                h[n] = abar * h[n] + bbar * x[i];
                acc += Ct[n] * h[n];
                if (h_all) h_all[((b * L + t) * Dn + d) * N + n] = h[n];
            }
            acc += (Dskip ? Dskip[d] : 0.0) * x[i];
            y[i] = z ? acc * silu(z[i]) : acc;
        }
        if (h_last)
            for (int64_t n = 0; n < N; ++n) h_last[(b * Dn + d) * N + n] = h[n];
        free(h);
    }
    return err;
}

/*
 * Speculative-decoding rollback (Algorithm 1: keep the verifier state at the
 * bifurcation). accept[s] = number of drafted bytes accepted on stream s, in
 * [0, k]. The kept state is h0[s] when nothing was accepted, otherwise the
 * state after the accept[s]-th drafted byte, h_all[s, accept[s]-1].
 */
int oracle_rollback(int64_t batch, int64_t k, int64_t Dn, int64_t N,
                    const double *h0, const double *h_all, const int32_t *accept,
                    double *h_out)
{
    int64_t per = Dn * N;
    for (int64_t s = 0; s < batch; ++s) {
        int32_t a = accept[s];
        if (a < 0 || a > k) return 1;
        const double *src = (a == 0) ? (h0 ? h0 + s * per : NULL)
                                     : h_all + (s * k + (a - 1)) * per;
        for (int64_t j = 0; j < per; ++j) h_out[s * per + j] = src ? src[j] : 0.0;
    }
    return 0;
}

/*
 * Backward of the layer core (training path: the paper trains through this
 * scan, Section 2 "parallel scans" and Section 4 training setup). Given the
 * forward inputs and the upstream gradients dout = dJ/dout [batch, L, D] and
 * dh_last = dJ/dh_last [batch, D, N] (NULL = 0), returns every input
 * gradient of J. Euler rule for B only (the path's rule).
 *
 * The adjoint recurrence, per (b, d), from t = L-1 down to 0, where
 * g[n] = dJ/dh_t[n] (starting from dh_last):
 *   s      = silu(z_t) (1 without a gate),   dy = dout_t * s
 *   dz_t   = dout_t * y_t * silu'(z_t),      y_t = sum_n C h_t + D x_t
 *   g[n]  += dy * C[t,n];     dC[t,n] += dy * h_t[n];     dD += dy * x_t
 *   S1     = sum_n g[n] B[t,n]
 *   dx_t   = dy * D + Delta_t * S1;          dDelta = x_t * S1
 *   dB[t,n] += g[n] * Delta_t * x_t
 *   w[n]   = g[n] * h_{t-1}[n] * Abar_t[n]   (dJ/dAbar times Abar)
 *   dDelta += sum_n w[n] A[n];  dA[n] += w[n] * Delta_t;  g[n] *= Abar_t[n]
 *   ddt_t  = dDelta * sigmoid(dt_t + bias);  dbias += ddt_t
 * and finally dh0 = g. dB, dC are summed over d; dA, dD, dbias over b and t.
 * Sums over channels are taken per thread and then added in thread order.
 */
static double sigmoid(double v) { return 1.0 / (1.0 + exp(-v)); }

int oracle_scan_backward(int64_t batch, int64_t L, int64_t Dn, int64_t N,
                         const double *x, const double *z, const double *dt,
                         const double *B, const double *C, const double *A,
                         const double *Dskip, const double *dt_bias, const double *h0,
                         const double *dout, const double *dh_last,
                         double *dx, double *dz, double *ddt, double *dB, double *dC,
                         double *dA, double *dD, double *ddt_bias, double *dh0,
                         int nthreads)
{
    if (batch < 0 || L < 0 || Dn < 0 || N <= 0) return 1;
    if (nthreads < 1) nthreads = 1;
    int64_t bl = batch * L * N;
    for (int64_t j = 0; j < bl; ++j) { dB[j] = 0.0; dC[j] = 0.0; }
    for (int64_t j = 0; j < Dn * N; ++j) dA[j] = 0.0;
    for (int64_t d = 0; d < Dn; ++d) { dD[d] = 0.0; ddt_bias[d] = 0.0; }
    double *partB = (double *)calloc((size_t)(nthreads * bl + 1), sizeof(double));
    double *partC = (double *)calloc((size_t)(nthreads * bl + 1), sizeof(double));
    if (!partB || !partC) { free(partB); free(partC); return 1; }
    int err = 0;
    /* one channel d (all batch rows) per iteration: dA, dD, dbias of d are
     * private to it; dB, dC go to per-thread partial sums */
#pragma omp parallel for num_threads(nthreads) schedule(dynamic, 1) reduction(| : err)
    for (int64_t d = 0; d < Dn; ++d) {
#ifdef _OPENMP
        int tid = omp_get_thread_num();
#else
        int tid = 0;
#endif
        double *pB = partB + (int64_t)tid * bl, *pC = partC + (int64_t)tid * bl;
        double *hh = (double *)malloc((size_t)((L + 1) * N) * sizeof(double)); /* h_{-1} .. h_{L-1} */
        double *ab = (double *)malloc((size_t)(L * N + 1) * sizeof(double));
        double *dl = (double *)malloc((size_t)(L + 1) * sizeof(double));
        double *yp = (double *)malloc((size_t)(L + 1) * sizeof(double));
        double *g = (double *)malloc((size_t)N * sizeof(double));
        if (!hh || !ab || !dl || !yp || !g) { err |= 1; free(hh); free(ab); free(dl); free(yp); free(g); continue; }
        double bias = dt_bias ? dt_bias[d] : 0.0, dsk = Dskip ? Dskip[d] : 0.0;
        for (int64_t b = 0; b < batch; ++b) {
            /* forward, keeping every state */
            for (int64_t n = 0; n < N; ++n) hh[n] = h0 ? h0[(b * Dn + d) * N + n] : 0.0;
            for (int64_t t = 0; t < L; ++t) {
                int64_t i = (b * L + t) * Dn + d;
                const double *Bt = B + (b * L + t) * N, *Ct = C + (b * L + t) * N;
                double delta = softplus(dt[i] + bias), acc = 0.0;
                dl[t] = delta;
                for (int64_t n = 0; n < N; ++n) {
                    double abar = exp(delta * A[d * N + n]);
                    ab[t * N + n] = abar;
                    hh[(t + 1) * N + n] = abar * hh[t * N + n] + delta * Bt[n] * x[i];
                    acc += Ct[n] * hh[(t + 1) * N + n];
                }
                yp[t] = acc + dsk * x[i];
            }
            /* backward */
            for (int64_t n = 0; n < N; ++n) g[n] = dh_last ? dh_last[(b * Dn + d) * N + n] : 0.0;
            for (int64_t t = L - 1; t >= 0; --t) {
                int64_t i = (b * L + t) * Dn + d;
                const double *Bt = B + (b * L + t) * N, *Ct = C + (b * L + t) * N;
                double dy = dout[i];
                if (z) {
                    double sz = sigmoid(z[i]);
                    dz[i] = dout[i] * yp[t] * sz * (1.0 + z[i] * (1.0 - sz));
                    dy = dout[i] * silu(z[i]);
                }
                dD[d] += dy * x[i];
                double S1 = 0.0;
                for (int64_t n = 0; n < N; ++n) {
                    g[n] += dy * Ct[n];
                    pC[(b * L + t) * N + n] += dy * hh[(t + 1) * N + n];
                    S1 += g[n] * Bt[n];
                }
                double delta = dl[t];
                dx[i] = dy * dsk + delta * S1;
                double ddelta = x[i] * S1;
                for (int64_t n = 0; n < N; ++n) {
                    pB[(b * L + t) * N + n] += g[n] * delta * x[i];
                    double w = g[n] * hh[t * N + n] * ab[t * N + n];
                    ddelta += w * A[d * N + n];
                    dA[d * N + n] += w * delta;
                    g[n] *= ab[t * N + n];
                }
                ddt[i] = ddelta * sigmoid(dt[i] + bias);
                ddt_bias[d] += ddt[i];
            }
            for (int64_t n = 0; n < N; ++n) dh0[(b * Dn + d) * N + n] = g[n];
        }
        free(hh); free(ab); free(dl); free(yp); free(g);
    }
    for (int th = 0; th < nthreads; ++th)
        for (int64_t j = 0; j < bl; ++j) {
            dB[j] += partB[(int64_t)th * bl + j];
            dC[j] += partC[(int64_t)th * bl + j];
        }
    free(partB); free(partC);
    return err;
}
