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
