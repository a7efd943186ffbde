/*
 * rikfad_oracle.c -- plain float64 CPU implementation of the Rank-1 iKFAD
 * (R-iKFAD) optimiser step, written to be checked by eye against the paper
 * ("Low-Rank Friction for Memory-Efficient Transformer Pretraining",
 * Rajpal & Leimkuhler), not to be fast.
 *
 * TEST INFRASTRUCTURE.  Only the test-suite, the smoke check and the CPU
 * baseline leg of the benchmark load this code.  The product library never
 * links, loads or calls it, and the two share no source, header, table or
 * helper.
 *
 * Conventions
 *   - Every value is IEEE float64.  exp/expm1 are the C library's.
 *   - A matrix parameter X is m x n, stored row-major (X[i*n + j]).  Rows are
 *     indexed by i (the factor R has m entries), columns by j (C has n).
 *   - Each sub-step of the BACD splitting is one plain loop over all
 *     elements, in the order the paper states them (Appendix A, Table
 *     "Analytical sub-step update rules"): B, A, C, D.  Intermediate momenta
 *     overwrite P in place; nothing is fused or reordered.
 *
 * Pins (tests/test_oracle_pins.py): every exported function is checked
 * against something other than itself -- the continuous dynamics integrated
 * by scipy (first-order convergence of the whole step, third-order local
 * error of sub-step C, exact factor filter), closed forms (heavy-ball /
 * symplectic-Euler recurrence, pure decay, rank-1 equivalence with
 * element-wise iKFAD), the paper's proved invariants, and the energy-decay
 * slopes the paper prints (Table "Local slopes of log E").  No function here
 * is parity-unpinned.
 */
#include <math.h>
#include <stdint.h>

/* Error codes returned by every entry point. */
#define ORC_OK 0
#define ORC_EARG (-1)

static int hparams_ok(double h, double alpha, double mu, double gamma, double eps_stab)
{
    /* Section 2 and Theorem 1: alpha, mu > 0, gamma >= 0, eps_stab >= 0
     * (eps_stab = 0 is the convention of Theorem 3).  mu = +inf is accepted:
     * it switches the friction forcing off, which the closed-form pins use. */
    return h >= 0.0 && alpha > 0.0 && mu > 0.0 && gamma >= 0.0 && eps_stab >= 0.0;
}

/* Sum of the row factor, 1_m^T R (denominator of Eq. xi_def). */
static double row_factor_total(int64_t m, const double *R)
{
    double s = 0.0;
    for (int64_t i = 0; i < m; ++i)
        s += R[i];
    return s;
}

/* Rank-1 friction entry, Eq. (xi_def):
 *   xi~_ij = R_i C_j / (1_m^T R + eps_stab),
 * with xi~ = 0 when the denominator is zero (eps_stab = 0 and R = 0; the
 * convention stated with Theorem 3 and in the numerical setup appendix). */
static double friction_entry(double Ri, double Cj, double denom)
{
    if (denom == 0.0)
        return 0.0;
    return Ri * Cj / denom;
}

/*
 * One BACD step of R-iKFAD for one matrix parameter (Appendix A, Table
 * "Analytical sub-step update rules"; continuous system Eqs. rikfad_x to
 * rikfad_C; splitting Phi_h = D o C o A o B in Section 2).
 *
 *   X, P  : m*n, row-major, updated in place to X_{n+1}, P_{n+1}
 *   R, C  : m and n, updated in place to R_{n+1}, C_{n+1}
 *   G     : m*n, the gradient grad f(X_n)
 *   h     : step size; alpha, mu, gamma, eps_stab: hyperparameters
 *   rowsq : scratch of m doubles, colsq: scratch of n doubles (caller-owned)
 *   P1    : NULL, or m*n doubles that receive the half-damped momentum P^(1)
 *           of sub-step C (an output only; nothing else depends on it)
 */
int orc_step_matrix(int64_t m, int64_t n, double *X, double *P, double *R, double *C,
                    const double *G, double h, double alpha, double mu, double gamma,
                    double eps_stab, double *rowsq, double *colsq, double *P1)
{
    /* m = 0 is an empty matrix: no momentum, and C only decays. */
    if (m < 0 || n < 1 || !hparams_ok(h, alpha, mu, gamma, eps_stab))
        return ORC_EARG;
    const int64_t N = m * n;

    /* Sub-step B, gradient kick: P^(B) = P_n - h grad f(X_n). */
    for (int64_t k = 0; k < N; ++k)
        P[k] = P[k] - h * G[k];

    /* Sub-step A, drift with the kicked momentum: X_{n+1} = X_n + h P^(B). */
    for (int64_t k = 0; k < N; ++k)
        X[k] = X[k] + h * P[k];

    /* Sub-step C, first half: friction of the current factors,
     * xi~_n = R_n C_n^T / (1^T R_n + eps_stab), and
     * P^(1) = P^(B) (.) exp(-(h/2) xi~_n). */
    double denom = row_factor_total(m, R) + eps_stab;
    for (int64_t i = 0; i < m; ++i)
        for (int64_t j = 0; j < n; ++j)
            P[i * n + j] = P[i * n + j] * exp(-0.5 * h * friction_entry(R[i], C[j], denom));
    if (P1 != 0)
        for (int64_t k = 0; k < N; ++k)
            P1[k] = P[k];

    /* Sub-step C, factor update with the momentum held at P^(1): the exact
     * solution over time h of dR/dt = [P]^2 1_n / mu - alpha R (and the same
     * for C with the column sums),
     *   R_{n+1} = e^{-alpha h} R_n + (1 - e^{-alpha h})/(mu alpha) [P^(1)]^2 1_n,
     *   C_{n+1} = e^{-alpha h} C_n + (1 - e^{-alpha h})/(mu alpha) ([P^(1)]^2)^T 1_m.
     * 1 - e^{-alpha h} is evaluated as -expm1(-alpha h) (same number, no
     * cancellation). */
    const double decay = exp(-alpha * h);
    const double gain = -expm1(-alpha * h) / (mu * alpha);
    for (int64_t i = 0; i < m; ++i)
        rowsq[i] = 0.0;
    for (int64_t j = 0; j < n; ++j)
        colsq[j] = 0.0;
    for (int64_t i = 0; i < m; ++i)
        for (int64_t j = 0; j < n; ++j) {
            const double q = P[i * n + j] * P[i * n + j];
            rowsq[i] += q;
            colsq[j] += q;
        }
    for (int64_t i = 0; i < m; ++i)
        R[i] = decay * R[i] + gain * rowsq[i];
    for (int64_t j = 0; j < n; ++j)
        C[j] = decay * C[j] + gain * colsq[j];

    /* Sub-step C, second half: friction of the updated factors,
     * P^(2) = P^(1) (.) exp(-(h/2) xi~_{n+1}). */
    denom = row_factor_total(m, R) + eps_stab;
    for (int64_t i = 0; i < m; ++i)
        for (int64_t j = 0; j < n; ++j)
            P[i * n + j] = P[i * n + j] * exp(-0.5 * h * friction_entry(R[i], C[j], denom));

    /* Sub-step D, linear damping: P_{n+1} = P^(2) e^{-gamma h} (the identity
     * when gamma = 0, R-iKFAD0). */
    const double damp = exp(-gamma * h);
    for (int64_t k = 0; k < N; ++k)
        P[k] = P[k] * damp;
    return ORC_OK;
}

/*
 * One BACD step of element-wise iKFAD for a parameter that is not a matrix
 * (biases, LayerNorm scales).  Section 2 ("Memory Complexity") says such
 * parameters reduce to element-wise iKFAD with one extra scalar each: the
 * friction xi has the parameter's shape and obeys Eqs. ikfad_1 to ikfad_3,
 *   dx/dt = p,  dp/dt = -grad f - (gamma + xi) (.) p,  dxi/dt = [p]^2/mu - alpha xi,
 * discretised with the same B, A, C, D sub-steps as the matrix case, xi
 * taking the place of xi~ and [P^(1)]^2 element-wise taking the place of its
 * row and column sums.
 *
 *   x, p, xi : L values, updated in place; g: L gradient values
 */
int orc_step_vector(int64_t L, double *x, double *p, double *xi, const double *g, double h,
                    double alpha, double mu, double gamma)
{
    if (L < 0 || !hparams_ok(h, alpha, mu, gamma, 0.0))
        return ORC_EARG;

    /* B */
    for (int64_t k = 0; k < L; ++k)
        p[k] = p[k] - h * g[k];
    /* A */
    for (int64_t k = 0; k < L; ++k)
        x[k] = x[k] + h * p[k];
    /* C, first half-damp with xi_n */
    for (int64_t k = 0; k < L; ++k)
        p[k] = p[k] * exp(-0.5 * h * xi[k]);
    /* C, exact filter of xi forced by the half-damped momentum */
    const double decay = exp(-alpha * h);
    const double gain = -expm1(-alpha * h) / (mu * alpha);
    for (int64_t k = 0; k < L; ++k)
        xi[k] = decay * xi[k] + gain * p[k] * p[k];
    /* C, second half-damp with xi_{n+1} */
    for (int64_t k = 0; k < L; ++k)
        p[k] = p[k] * exp(-0.5 * h * xi[k]);
    /* D */
    const double damp = exp(-gamma * h);
    for (int64_t k = 0; k < L; ++k)
        p[k] = p[k] * damp;
    return ORC_OK;
}

/*
 * Energy of Section 3 (Eq. energy of the rates appendix) for the quadratic
 * f(X) = 1/2 vec(X)^T A vec(X) with dense symmetric A (d x d, d = m n), whose
 * minimiser is X* = 0 with f* = 0:
 *   E = 1/2 vec(X)^T A vec(X) + 1/2 ||P||_F^2.
 */
double orc_dense_quadratic_energy(int64_t d, const double *A, const double *x, const double *p)
{
    double quad = 0.0, kin = 0.0;
    for (int64_t a = 0; a < d; ++a) {
        double Ax = 0.0;
        for (int64_t b = 0; b < d; ++b)
            Ax += A[a * d + b] * x[b];
        quad += x[a] * Ax;
        kin += p[a] * p[a];
    }
    return 0.5 * quad + 0.5 * kin;
}

/*
 * BACD integration of R-iKFAD on f(X) = 1/2 vec(X)^T A vec(X), the test
 * problem of the numerical-validation section (Section 3.2 and the
 * numerical-setup appendix): grad f(X) = A vec(X), reshaped m x n.
 *
 *   X, P (m*n), R (m), C (n) : initial state, advanced in place
 *   nsteps                   : number of steps of size h
 *   record, nrecord          : ascending step indices k (0 <= k <= nsteps) at
 *                              which E(t = k h) is written to energy[]
 *   work                     : scratch of m*n + m + n doubles
 * Returns 0, or -1 on a bad argument.
 */
int orc_dense_quadratic_run(int64_t m, int64_t n, const double *A, double *X, double *P,
                            double *R, double *C, double h, double alpha, double mu,
                            double gamma, double eps_stab, int64_t nsteps,
                            const int64_t *record, int64_t nrecord, double *energy,
                            double *work)
{
    if (m < 1 || n < 1 || nsteps < 0 || nrecord < 0)
        return ORC_EARG;
    const int64_t d = m * n;
    double *G = work, *rowsq = work + d, *colsq = work + d + m;
    int64_t next = 0;
    for (int64_t k = 0; k <= nsteps; ++k) {
        while (next < nrecord && record[next] == k) {
            energy[next] = orc_dense_quadratic_energy(d, A, X, P);
            ++next;
        }
        if (k == nsteps)
            break;
        for (int64_t a = 0; a < d; ++a) {
            double g = 0.0;
            for (int64_t b = 0; b < d; ++b)
                g += A[a * d + b] * X[b];
            G[a] = g;
        }
        int rc = orc_step_matrix(m, n, X, P, R, C, G, h, alpha, mu, gamma, eps_stab, rowsq,
                                 colsq, 0);
        if (rc != ORC_OK)
            return rc;
    }
    return next == nrecord ? ORC_OK : ORC_EARG;
}
