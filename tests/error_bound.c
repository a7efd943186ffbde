/*
 * error_bound.c -- first-order bound on how far the float32 step kernels may
 * lie from the float64 oracle, per element, carried along an oracle
 * trajectory.  TEST INFRASTRUCTURE: it models the rounding of the kernels'
 * arithmetic (every float32 operation correctly rounded, relative error at
 * most U = 2^-24; exp2f within 2 ulp, i.e. 4U relative); it is neither the
 * oracle nor the kernels, and computes no expected value.
 *
 * One step of the matrix rule (Appendix A of the paper: B, A, C, D), as the
 * kernels evaluate it for element (i, j):
 *   p_n  = (p^ e_prev) damp_prev        the canonical momentum P_n
 *   p_b  = fma(-h, g, p_n)              B  (h rounded to float32)
 *   x'   = fma(h, p_b, x)               A
 *   p1   = p_b exp(-z0)                 C, first half-damp, z0 = (h/2) xi~_n
 *   P'   = p1 exp(-z1) e^{-gamma h}     C second half-damp and D (the next
 *                                       step's p_n, or the canonical output),
 *                                       z1 = (h/2) xi~_{n+1}
 * With EP the bound on |p_n - P_n| and EX on |x - X_n|, first order:
 *   E_pb  = EP + U (|P^(B)| + 2 h |g|)               (rounding of h and of the fma)
 *   EX'   = EX + h E_pb + U (|X_{n+1}| + 2 h |P^(B)|)
 *   E_p1  = E_pb + |P^(1)| (5U + Ez0)               (exp2f 4U, product U, argument Ez0)
 *   EP'   = E_p1 + |P_{n+1}| (7U + Ez1)             (exp2f 4U, two products and e^{-gamma h}
 *                                                    rounded to float32 3U; damping <= 1
 *                                                    carries E_p1 at most whole)
 * where Ez is the error of the exponent: (h/2) (dR_i C_j + R_i dC_j)/(s + eps)
 * + z (ds/(s + eps) + 6U) (six roundings: -(h/2) log2 e, s + eps, its
 * reciprocal, R_i times it, the scale, C_j times that), dR and dC the
 * deviations of the factors the
 * kernel used (measured by the caller, and compared with the oracle by the
 * tests themselves), ds that of 1^T R.  The terms U |P^(B)| + 2U h |g| and
 * U |X_{n+1}| + 2U h |P^(B)| are the cancellation scales: where P_n and h g
 * (or X_n and h P^(B)) nearly cancel, the result is tiny but its error is a
 * rounding of the larger terms.  The factors' bound (used only where a factor
 * misses the pure relative tolerance, e.g. a one-column matrix whose R_i is a
 * single square) is, given the previous deviation dR:
 *   ER_i = d dR_i + k sum_j (2 |P^(1)_ij| E_p1 + E_p1^2) + (depth_row + 4) U R_i
 * (|P^(1)| is bounded by |P^(B)| throughout, since the friction only damps)
 * and likewise EC_j, with the summation depths of the kernels' row and column
 * sums supplied by the caller.
 *
 * Element-wise rule: the same B and A; the friction xi is filtered from the
 * element's own square, xi' = d xi + k [P^(1)]^2 (one fma), so its bound is
 * carried per element: Exi' = d Exi + k (2 |P^(1)| E_p1 + E_p1^2) + 5U xi',
 * with Ez = (h/2) Exi + 2U z.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>

static const double U = 1.0 / 16777216.0;

static double inv_den(double s, double eps)
{
    const double den = s + eps;
    return den == 0.0 ? 0.0 : 1.0 / den;
}

/* Matrix rule, one step.  Oracle arrays (row-major, double): X0, P0 (P
 * canonical) before the step, G the gradient, X1, P1 after; R0, C0 / R1, C1
 * the oracle's factors before / after; dR0, dC0 / dR1, dC1 the measured
 * |kernel - oracle| deviations of those factors (NULL: zero).  EX, EP are
 * carried (in/out); ER, EC receive the factors' bound after the step, and
 * EP1 (unless NULL) that of the half-damped momentum P^(1) (the stored form).
 * Returns 0, or -1 if a work array cannot be allocated. */
int eb_matrix_step(int64_t m, int64_t n, double h, double eps, double decay, double gain,
                   const double *X0, const double *P0, const double *G, const double *X1,
                   const double *P1, const double *R0, const double *C0, const double *R1,
                   const double *C1, const double *dR0, const double *dC0, const double *dR1,
                   const double *dC1, double depth_row, double depth_col, double *EX, double *EP,
                   double *ER, double *EC, double *EP1)
{
    double s0 = 0.0, s1 = 0.0, ds0 = 0.0, ds1 = 0.0;
    for (int64_t i = 0; i < m; ++i) {
        s0 += R0[i];
        s1 += R1[i];
        ds0 += dR0 ? dR0[i] : 0.0;
        ds1 += dR1 ? dR1[i] : 0.0;
    }
    /* 1^T R: trees over 256 rows (8 levels), then the partial sums added
     * lane by lane (m / 8192 each) and a 32-lane tree (5 levels) */
    const double sum_depth = 16.0 + (double)(m / 8192) + 8.0;
    ds0 += sum_depth * U * s0;
    ds1 += sum_depth * U * s1;
    const double i0 = inv_den(s0, eps), i1 = inv_den(s1, eps);
    double *colacc = (double *)calloc((size_t)(n > 0 ? n : 1), sizeof(double));
    if (colacc == NULL)
        return -1;
    for (int64_t i = 0; i < m; ++i) {
        double rowacc = 0.0;
        for (int64_t j = 0; j < n; ++j) {
            const int64_t a = i * n + j;
            const double z0 = 0.5 * h * R0[i] * C0[j] * i0;
            const double z1 = 0.5 * h * R1[i] * C1[j] * i1;
            const double ez0 = 0.5 * h * ((dR0 ? dR0[i] : 0.0) * C0[j] + R0[i] * (dC0 ? dC0[j] : 0.0)) * i0 +
                               z0 * (ds0 * i0 + 6.0 * U);
            const double ez1 = 0.5 * h * ((dR1 ? dR1[i] : 0.0) * C1[j] + R1[i] * (dC1 ? dC1[j] : 0.0)) * i1 +
                               z1 * (ds1 * i1 + 6.0 * U);
            const double hg = h * fabs(G[a]);
            const double pb = fabs(P0[a] - h * G[a]);
            const double epb = EP[a] + U * (pb + 2.0 * hg);
            EX[a] += h * epb + U * (fabs(X1[a]) + 2.0 * h * pb);
            const double p1 = pb;           /* |P^(1)| <= |P^(B)|: the friction only damps */
            const double ep1 = epb + p1 * (5.0 * U + ez0);
            const double q = 2.0 * p1 * ep1 + ep1 * ep1;
            rowacc += q;
            colacc[j] += q;
            if (EP1)
                EP1[a] = ep1;
            EP[a] = ep1 + fabs(P1[a]) * (7.0 * U + ez1);
        }
        ER[i] = decay * (dR0 ? dR0[i] : 0.0) + gain * rowacc + (depth_row + 4.0) * U * R1[i];
    }
    for (int64_t j = 0; j < n; ++j)
        EC[j] = decay * (dC0 ? dC0[j] : 0.0) + gain * colacc[j] + (depth_col + 4.0) * U * C1[j];
    free(colacc);
    return 0;
}

/* Element-wise rule, one step, L elements: oracle X0, P0, XI0 before, G,
 * X1, P1, XI1 after; EX, EP, EXI carried (in/out). */
void eb_vector_step(int64_t L, double h, double decay, double gain, const double *X0,
                    const double *P0, const double *XI0, const double *G, const double *X1,
                    const double *P1, const double *XI1, double *EX, double *EP, double *EXI)
{
    for (int64_t a = 0; a < L; ++a) {
        const double z0 = 0.5 * h * XI0[a];
        const double ez0 = 0.5 * h * EXI[a] + 2.0 * U * z0;
        const double hg = h * fabs(G[a]);
        const double pb = fabs(P0[a] - h * G[a]);
        const double epb = EP[a] + U * (pb + 2.0 * hg);
        EX[a] += h * epb + U * (fabs(X1[a]) + 2.0 * h * pb);
        const double p1 = pb;               /* |P^(1)| <= |P^(B)| */
        const double ep1 = epb + p1 * (5.0 * U + ez0);
        EXI[a] = decay * EXI[a] + gain * (2.0 * p1 * ep1 + ep1 * ep1) + 5.0 * U * XI1[a];
        const double z1 = 0.5 * h * XI1[a];
        const double ez1 = 0.5 * h * EXI[a] + 2.0 * U * z1;
        EP[a] = ep1 + fabs(P1[a]) * (7.0 * U + ez1);
    }
}
