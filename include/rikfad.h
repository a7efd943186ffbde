/*
 * rikfad.h -- C ABI of the GB300 (sm_103a) Rank-1 iKFAD (R-iKFAD) optimiser.
 *
 * R-iKFAD ("Low-Rank Friction for Memory-Efficient Transformer Pretraining",
 * Rajpal & Leimkuhler) is momentum descent with an adaptive friction.  For a
 * matrix parameter X (m x n) it keeps the full momentum P and two factors
 * R (m) and C (n) whose outer product gives the friction
 *     xi~_ij = R_i C_j / (1_m^T R + eps_stab)                       (Eq. xi_def)
 * (Section 2, Eqs. rikfad_x to rikfad_C).  One optimiser step is the BACD
 * splitting of Appendix A (Table "Analytical sub-step update rules"):
 *     B  P^(B) = P_n - h grad f(X_n)
 *     A  X_{n+1} = X_n + h P^(B)
 *     C  P^(1) = P^(B) (.) exp(-(h/2) xi~_n)
 *        R_{n+1} = e^{-alpha h} R_n + (1 - e^{-alpha h})/(mu alpha) [P^(1)]^2 1_n
 *        C_{n+1} = e^{-alpha h} C_n + (1 - e^{-alpha h})/(mu alpha) ([P^(1)]^2)^T 1_m
 *        P^(2) = P^(1) (.) exp(-(h/2) xi~_{n+1})
 *     D  P_{n+1} = P^(2) e^{-gamma h}
 * Parameters that are not matrices (biases, LayerNorm) follow element-wise
 * iKFAD (Section 2, "Memory Complexity"): a friction scalar per element
 * takes the place of xi~ and is filtered from its own [P^(1)]^2.
 *
 * Conventions for every call:
 *   - Pointers named "device" are CUDA device pointers of the device that was
 *     current when the handle was created; "host" pointers are CPU memory.
 *   - Tensors are dense and row-major.  A matrix (rows m, cols n) element
 *     (i, j) is at offset i*n + j.  Parameters and momenta are float32;
 *     gradients are float32 or bfloat16, fixed per handle.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream).  Work is enqueued on it and nothing waits on the host unless the
 *     call says so.  The library never synchronises the device.
 *   - Every call that can fail returns a rikfad_status; on failure
 *     rikfad_last_error() describes it (thread-local string).  Argument errors
 *     are detected before any work is enqueued.  Errors of work already
 *     enqueued surface as RIKFAD_ERR_CUDA on a later call.
 *   - A handle is not thread-safe: calls on one handle must not overlap.
 *     Its device work shares the handle's workspace and state, so it must
 *     also be ordered on the GPU: enqueue it on one stream, or order the
 *     streams with events.
 *   - Non-finite guard.  The friction of Eq. xi_def divides by 1^T R +
 *     eps_stab and every element of a matrix reads R and C, so one
 *     non-finite gradient or momentum element poisons its whole matrix
 *     within a step (and, with the paper's GPT2-S setting mu = 1.36e-6, the
 *     gain (1 - e^{-alpha h})/(mu alpha) ~ 7e4 amplifies any blow-up).  The
 *     kernels therefore test every R_i and C_j they write, every partial sum
 *     of 1^T R and every element-wise friction value; a non-finite one is
 *     recorded on the device and in a page-locked host flag.  A non-finite
 *     P^(1) always shows there (R_i sums its row's squares, C_j its
 *     column's); a non-finite X alone (a caller-supplied one, with finite
 *     momentum) does not.  Once a report is visible on the host, rikfad_step
 *     returns RIKFAD_ERR_NONFINITE and enqueues nothing; rikfad_check_finite
 *     waits, names the tensor and clears the report.  The check adds no
 *     memory traffic.
 */
#ifndef RIKFAD_H
#define RIKFAD_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#if defined(__GNUC__)
#define RIKFAD_API __attribute__((visibility("default")))
#else
#define RIKFAD_API
#endif

/* Status codes. */
enum rikfad_status {
    RIKFAD_OK = 0,
    RIKFAD_ERR_ARG = -1,   /* null pointer, bad shape, bad hyperparameter, bad index */
    RIKFAD_ERR_ALIGN = -2, /* a pointer does not meet the documented alignment */
    RIKFAD_ERR_CUDA = -3,  /* a CUDA runtime call or an earlier kernel failed */
    RIKFAD_ERR_OOM = -4,   /* device or pinned host allocation failed */
    RIKFAD_ERR_NONFINITE = -5, /* a step produced a non-finite factor, friction or 1^T R */
    RIKFAD_ERR_STATE = -6  /* call not valid for this handle (e.g. wrong device) */
};

/* Gradient element type, fixed per handle. */
enum rikfad_grad_dtype { RIKFAD_GRAD_F32 = 0, RIKFAD_GRAD_BF16 = 1 };

/* Hyperparameters of Eqs. rikfad_x to rikfad_C and Eq. xi_def: the factor
 * decay alpha > 0, the friction scale mu > 0, the linear damping gamma >= 0
 * (gamma = 0 is R-iKFAD0, the paper's default, Section 4.2) and the
 * stabiliser eps_stab >= 0 (the paper fixes 1e-16, Section 4).  With
 * eps_stab = 0 the friction is zero while 1^T R = 0 (Theorem 3's convention). */
typedef struct {
    double alpha;
    double mu;
    double gamma;
    double eps_stab;
} rikfad_hparams;

/* Shape of one parameter tensor.  cols >= 1: an m x n matrix (rows = m >= 0)
 * with factors R (m) and C (n).  cols == 0: a tensor that is not a matrix,
 * flattened to `rows` >= 0 elements, updated element-wise. */
typedef struct {
    int64_t rows;
    int64_t cols;
} rikfad_shape;

typedef struct rikfad_handle_s *rikfad_handle;

/*
 * Create an optimiser for a fixed list of parameter tensors on the current
 * CUDA device.  Allocates and zeroes the factors R, C and the element-wise
 * friction (R(0) = C(0) = 0, as in Lemma 1 and the numerical appendix), plus
 * the reduction workspace, and plans the fused kernels for this list.
 *   shapes     host array of `ntensors` shapes (ntensors >= 0), copied
 *   hp         host pointer, copied; alpha, mu > 0, gamma, eps_stab >= 0
 *   grad_dtype RIKFAD_GRAD_F32 or RIKFAD_GRAD_BF16
 *   out        receives the handle (NULL on failure)
 * Errors: RIKFAD_ERR_ARG, RIKFAD_ERR_OOM, RIKFAD_ERR_CUDA.
 */
RIKFAD_API int rikfad_create(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp,
                             int grad_dtype, rikfad_handle *out);

/*
 * Create a full-friction iKFAD optimiser (the method R-iKFAD factorises,
 * Eqs. ikfad_1 to ikfad_3): every tensor, matrix or not, keeps one friction
 * scalar per element and follows the element-wise rule; the auxiliary state
 * is 2N floats (the iKFAD column of the paper's memory table).  Same handle
 * type, step, checkpoint and query calls as rikfad_create; rikfad_get_factors
 * returns a tensor's rows x cols friction values in R_host.  Every pointer
 * must be 16-byte aligned.  Errors as for rikfad_create.
 */
RIKFAD_API int rikfad_create_ikfad(const rikfad_shape *shapes, int ntensors, const rikfad_hparams *hp,
                                   int grad_dtype, rikfad_handle *out);

/*
 * Create full iKFAD with R-iKFAD's factors carried along as shadows: every
 * matrix keeps its element-wise friction xi (rows x cols floats) and steps by
 * full iKFAD, while its R and C follow R-iKFAD's factor filter from the same
 * half-damped momentum without being used in the update.  This is the set-up
 * of the paper's Section 4.4 ("How close is xi~ to the best rank-1
 * friction?"), read out by rikfad_friction_diagnostics.  Non-matrices follow
 * the element-wise rule as usual.  Same step and query calls as
 * rikfad_create; momenta are always canonical (no pending factor).  Every
 * pointer of a matrix whose cols is a multiple of 8 must be 16-byte aligned.
 */
RIKFAD_API int rikfad_create_ikfad_shadow(const rikfad_shape *shapes, int ntensors,
                                          const rikfad_hparams *hp, int grad_dtype,
                                          rikfad_handle *out);

/* Release the handle and everything it allocated (after a device sync of its
 * own work).  NULL is accepted. */
RIKFAD_API void rikfad_destroy(rikfad_handle h);

/*
 * Enqueue one R-iKFAD step of size `step` (> 0, finite) over every tensor.
 *   x[t]    device, float32, tensor t's parameters; updated to X_{n+1}
 *   grad[t] float32 or bfloat16 (per handle), grad f(X_n); read only.  Device
 *           memory, or page-locked host memory that the device can address
 *           (e.g. from cudaHostAlloc): the kernel then reads the gradient
 *           over the CPU-GPU link, with no separate copy
 *   p[t]    device, float32, tensor t's momentum in the library's stored form
 *           (below); updated
 * The three arrays are host arrays of `ntensors` device pointers, in the
 * order of the shapes given to rikfad_create; they may change from call to
 * call (a change costs one small host-to-device copy).  Every pointer must be
 * 16-byte aligned, except for matrices whose cols is not a multiple of 8 and
 * for which only natural alignment is required.  Pointers of empty tensors
 * may be NULL.  x, grad and p must not overlap.  When a pointer differs from
 * the previous call's, the host checks that the device can address it
 * (RIKFAD_ERR_ARG for memory of another device, or for pageable host memory
 * on a device that cannot read it through the host's page tables).
 *
 * Stored form of the momentum of a matrix: between steps p holds P^(1) of
 * the last step (the half-damped momentum) and the library remembers the
 * pending factor exp(-(h/2) xi~_{n+1}) e^{-gamma h} of sub-steps C and D,
 * which the next step applies on the fly (the values are identical to the
 * paper's P_{n+1}).  rikfad_materialize / rikfad_canonical_momentum give the
 * paper's P_{n+1}.  Element-wise tensors always hold P_{n+1}.  Before the
 * first step p must hold the initial momentum (normally zeros).
 */
RIKFAD_API int rikfad_step(rikfad_handle h, double step, float *const *x, const void *const *grad,
                           float *const *p, void *stream);

/*
 * Turn the stored momenta into the paper's P_{n+1} in place and clear the
 * pending factor, so the next step starts from canonical momenta.  Use before
 * checkpointing the momenta or handing them to other code.
 *   p  host array of ntensors device pointers (same rules as rikfad_step)
 */
RIKFAD_API int rikfad_materialize(rikfad_handle h, float *const *p, void *stream);

/*
 * Write the paper's P_{n+1} of every matrix into `out` without changing the
 * optimiser's state (the stored momenta and pending factor are left as they
 * are).  Element-wise tensors are copied.  out[t] must not overlap p[t].
 */
RIKFAD_API int rikfad_canonical_momentum(rikfad_handle h, const float *const *p,
                                         float *const *out, void *stream);

/* Optimiser auxiliary state in bytes, as counted in the paper's memory table
 * (Appendix "Memory Analysis"): factors R and C of every matrix plus the
 * element-wise friction (4 bytes each), plus, if include_momentum != 0, the
 * float32 momentum of every parameter.  Workspace is not included. */
RIKFAD_API size_t rikfad_state_bytes(rikfad_handle h, int include_momentum);

/* Same count for a shape list, without a handle or a GPU. */
RIKFAD_API size_t rikfad_state_bytes_for(const rikfad_shape *shapes, int ntensors,
                                         int include_momentum);

/* Device bytes the handle allocated besides the state (reduction partials,
 * plan tables, pointer table). */
RIKFAD_API size_t rikfad_workspace_bytes(rikfad_handle h);

/* The step size whose pending factor the stored momenta still carry (0 after
 * creation, rikfad_materialize or rikfad_import_state of a materialised
 * state). */
RIKFAD_API double rikfad_pending_step(rikfad_handle h);

/*
 * Copy tensor t's factors to the host (synchronises the device).
 * Matrix: R_host receives rows floats, C_host cols floats (either may be NULL).
 * Element-wise tensor: R_host receives its rows friction values; C_host unused.
 */
RIKFAD_API int rikfad_get_factors(rikfad_handle h, int t, float *R_host, float *C_host);

/* Overwrite tensor t's factors from the host (same layout as
 * rikfad_get_factors; values must be finite and >= 0).  Synchronises. */
RIKFAD_API int rikfad_set_factors(rikfad_handle h, int t, const float *R_host, const float *C_host);

/* Copy tensor t's element-wise friction to the host (synchronises): the
 * rows floats of a non-matrix, or the rows x cols floats (row-major) of a
 * matrix of a shadow handle.  RIKFAD_ERR_ARG for a matrix with rank-1
 * friction (its state is R and C, rikfad_get_factors). */
RIKFAD_API int rikfad_get_friction(rikfad_handle h, int t, float *xi_host);

/*
 * Friction diagnostics of matrix t of a shadow handle (rikfad_create_ikfad_
 * shadow), after the work enqueued on `stream` (synchronises).  Writes six
 * doubles to out (host):
 *   out[0]  ||xi - xi~||_F / ||xi||_F, xi~ = R C^T / (1^T R + eps_stab) from
 *           the shadow factors (the error of R-iKFAD's construction)
 *   out[1]  sqrt(1 - sigma_1^2 / ||xi||_F^2), the smallest relative error of
 *           any rank-1 approximation (Eckart-Young)
 *   out[2]  ||xi||_F^2 / sigma_1^2, the stable rank of xi
 *   out[3]  sigma_1, by power iteration on xi^T xi started from C, stopped
 *           when the estimate of sigma_1^2 changes by at most tol (relative)
 *           or after max_iters iterations
 *   out[4]  ||xi||_F
 *   out[5]  iterations used
 * All zeros for an all-zero friction.  RIKFAD_ERR_STATE for other handles.
 */
RIKFAD_API int rikfad_friction_diagnostics(rikfad_handle h, int t, int max_iters, double tol, double *out,
                                           void *stream);

/* Read the friction denominators 1^T R of every matrix (ntensors floats, 0 for
 * element-wise tensors) into host memory, enqueued on `stream`; the values
 * are valid once the stream reaches this point (the call itself waits for it).
 * Returns RIKFAD_ERR_NONFINITE (after writing host_out) if a step reported a
 * non-finite result; the report stays until rikfad_check_finite clears it. */
RIKFAD_API int rikfad_read_denominators(rikfad_handle h, float *host_out, void *stream);

/* The same read-back, enqueued only: the denominators kernel and a copy of
 * the ntensors floats into host_out are enqueued on `stream` and the call
 * returns at once, so a training loop can read step n's values while step
 * n + 1 runs (wait on the stream, or an event recorded after this call,
 * before reading host_out).  host_out: host memory the caller owns, page-locked
 * (cudaHostAlloc or cudaHostRegister) for the read-back to run asynchronously;
 * when it is mapped into the device's address space the kernel stores there
 * directly, otherwise a copy follows the kernel.  It must stay valid until
 * the stream has passed this point.  Non-finite results are reported by
 * rikfad_check_finite, not by this call. */
RIKFAD_API int rikfad_enqueue_denominators(rikfad_handle h, float *host_out, void *stream);

/*
 * Checkpoint support.  The state image is rikfad_state_image_bytes(h) bytes:
 * a 64-byte header (format tag, tensor count, pending step) followed by
 * every factor and element-wise friction value.  Momenta are not included
 * (the caller owns them; they are in the stored form of rikfad_step).
 *   export: dev_dst, device, receives the image (enqueued on stream)
 *   import: dev_src, device, an image exported by a handle with the same
 *           shapes and hyperparameters; synchronises to validate the header
 */
RIKFAD_API size_t rikfad_state_image_bytes(rikfad_handle h);
RIKFAD_API int rikfad_export_state(rikfad_handle h, void *dev_dst, void *stream);
RIKFAD_API int rikfad_import_state(rikfad_handle h, const void *dev_src, void *stream);

/*
 * Kernel timing.  While enabled, rikfad_step records CUDA events on its
 * stream around the fused step kernel and around the factor-finalise
 * kernel.  rikfad_profile_read waits for the recorded events and returns the
 * summed durations in milliseconds and the number of steps recorded since the
 * last enable; it then forgets them.
 */
RIKFAD_API int rikfad_profile_enable(rikfad_handle h, int enable);
RIKFAD_API int rikfad_profile_read(rikfad_handle h, double *step_kernel_ms,
                                   double *finalize_kernel_ms, int64_t *steps);

/*
 * Wait for the work enqueued on `stream` and report whether any step since
 * the last clear produced a non-finite factor R_i, C_j, partial sum of 1^T R
 * or element-wise friction value (the guard described at the top of this
 * header).  Returns RIKFAD_OK, or RIKFAD_ERR_NONFINITE with the lowest
 * offending tensor index in rikfad_last_error; in that case the report is
 * cleared, so that rikfad_step accepts work again once the caller has
 * restored a finite state (rikfad_import_state or rikfad_set_factors clear
 * the report as well).  The non-finite values themselves stay in the state.
 */
RIKFAD_API int rikfad_check_finite(rikfad_handle h, void *stream);

/* Number of kernel launches one rikfad_step enqueues for this handle. */
RIKFAD_API int rikfad_launches_per_step(rikfad_handle h);

/*
 * Work plan for a shape list, computed on the host for `nctas` blocks (no GPU
 * needed; the same planner rikfad_create uses).  Writes at most `cap` rows of
 * 8 int64 values into `out` (host) and returns the number of rows the plan
 * has (so a call with cap = 0 sizes the buffer), or a negative status.  Row:
 *   { block, tensor, kind (0 matrix rows, 1 element range), col0, width,
 *     begin, end, slot }
 * For kind 0 the block updates rows [begin, end) x columns [col0, col0+width)
 * of the matrix and writes its column partial sums to `slot`; for kind 1 it
 * updates elements [begin, end).
 */
RIKFAD_API int64_t rikfad_plan_query(const rikfad_shape *shapes, int ntensors, int grad_dtype,
                                     int nctas, int64_t *out, int64_t cap);

/*
 * Allocation-free step for one matrix.  This entry point has no counterpart
 * in the paper; it is a convenience of this library.
 *
 * rikfad_create allocates the factors and a reduction workspace with
 * cudaMalloc.  Some callers cannot allocate device memory on their own: a
 * framework whose caching allocator already holds the GPU's memory (a second
 * allocator next to it fails or fragments the pool), or a latency-bound
 * service that allows no cudaMalloc after start-up because the call can
 * synchronise the device and stall all its streams.  This call allocates
 * nothing: the caller owns every input and output, and the partial sums live
 * in a fixed 1.51 MB array compiled into the library, which every GPU that
 * loads the library keeps until the process exits.
 *
 * It performs one rikfad_step on a single matrix in the same stored form:
 *   rows, cols    0 <= rows <= 65536, 1 <= cols <= 1024 (anything larger is
 *                 rejected with RIKFAD_ERR_ARG)
 *   step          step size h > 0
 *   pending_step  the step size of this matrix's previous call (0 for the
 *                 first call, or after the momentum was made canonical);
 *                 the caller keeps this number, the library keeps no state
 *   hp            hyperparameters, as for rikfad_create
 *   grad_dtype    RIKFAD_GRAD_F32 or RIKFAD_GRAD_BF16
 *   x, grad, p    device, rows x cols row-major, as for rikfad_step (16-byte
 *                 aligned when cols is a multiple of 8)
 *   R, C          device, rows and cols floats: the factors, read and updated
 *                 (start them at zero)
 * The first call on each device looks up the array's device address (and
 * may load the library's device code onto that GPU); make that first call
 * before any stream capture.  A call enqueues three kernels on `stream` and
 * writes every partial sum before it reads it, so nothing in the array needs
 * to start at zero and calls in sequence are independent.  All calls share
 * the one array: calls whose work overlaps on the GPU (unordered streams)
 * race and give wrong results.  This call has no non-finite report (it has
 * no handle to keep one).  Errors as for rikfad_step, reported through
 * rikfad_last_error.
 */
RIKFAD_API int rikfad_step_matrix_noalloc(int64_t rows, int64_t cols, double step,
                                          double pending_step, const rikfad_hparams *hp,
                                          int grad_dtype, float *x, const void *grad, float *p,
                                          float *R, float *C, void *stream);

/*
 * Batched BACD integration of R-iKFAD on small dense quadratics (the test
 * problem of the paper's numerical validation of the gamma = 0 rates,
 * Section 3.2 and Table tab:g0_slopes): for every system s of the batch,
 *   f_s(X) = 1/2 vec(X)^T A_s vec(X),  grad f_s = A_s vec(X) reshaped m x n,
 * vec(X) row-major (element a = i n + j), and nsteps steps of size h of the
 * splitting of Appendix A (B, A, C, D in that order, the factors R (m) and
 * C (n) updated from the half-damped momentum), in float32.  Damping is
 * carried so that it survives when one step's damping is below float32
 * resolution of P (late in long gamma = 0 runs): P_k is formed only for the
 * energies and the output, and 1^T R is filtered alongside R from the total
 * of [P^(1)]^2 (equal to the sum of R up to rounding).
 *
 *   batch         number of systems, 0 <= batch <= 2^24 (0 does nothing)
 *   m, n          shape of every system: m >= 1, n >= 1, m n <= 32
 *   A             device, batch x (m n) x (m n) floats, row-major per system
 *                 (read only; the method needs no symmetry, the energy
 *                 below is the paper's only for symmetric A)
 *   X, P          device, batch x (m n) floats: position and the paper's
 *                 momentum P_k, read and advanced in place to the state
 *                 after nsteps steps
 *   R, C          device, batch x m and batch x n floats: the factors, read
 *                 and advanced in place (start them at zero, as the paper)
 *   step          h > 0;  hp as for rikfad_create (gamma enters as D)
 *   nsteps        number of steps, >= 0
 *   record        device, nrecord int64 step indices, strictly ascending;
 *                 for every record[r] in [0, nsteps] the energy
 *                 E = 1/2 vec(X)^T A vec(X) + 1/2 |P|_F^2 of the state after
 *                 record[r] steps is written to energy[r * batch + s].  Other
 *                 entries are skipped and their energies left untouched; a
 *                 list out of order loses the entries after the first descent.
 *   energy        device, nrecord x batch floats (written)
 * The call is asynchronous on `stream`.  It runs the steps in launches of S
 * steps from its start (S = 65536 for batch <= 32768, a smaller power of two
 * >= 128 for larger batches, so that no launch runs long); every launch
 * starts from the stored X, P, R, C.  A run split into consecutive calls at
 * a multiple of S (the second starting from the first's outputs, its record
 * indices counted from its own start) is therefore bit-identical to one
 * call; a split elsewhere agrees to float32 rounding.  Errors:
 * RIKFAD_ERR_ARG for sizes or hyperparameters out of range or a NULL pointer
 * that is needed, RIKFAD_ERR_ALIGN for a pointer not aligned to its element
 * type, RIKFAD_ERR_CUDA for a launch failure; messages via rikfad_last_error.
 */
RIKFAD_API int rikfad_quadratic_run(int64_t batch, int64_t m, int64_t n, const float *A, float *X,
                                    float *P, float *R, float *C, double step,
                                    const rikfad_hparams *hp, int64_t nsteps,
                                    const int64_t *record, int64_t nrecord, float *energy,
                                    void *stream);

/*
 * Testing hooks.  These have no counterpart in the paper.
 *
 * rikfad_debug_check_failures: a library compiled with -DRIKFAD_CHECKED
 * (librikfad_checked.so, built by build(checked=True)) verifies inside every
 * kernel of the default schedule (step, finalise, canonical momentum,
 * denominators), before each access, that the plan's block, piece, tensor, panel,
 * slot and finalise-item indices, the row, column and element ranges, the
 * offsets into the factor, partial-sum and denominator buffers, and the
 * pointer-table entries (non-NULL; 16-byte aligned on the 8-wide paths) lie
 * within what the planner produced.  A failed check is counted and the
 * access it guarded is skipped; nothing traps.  This call waits for the
 * device and writes the number of failed checks since the handle was created
 * to *count (and the code of the first, rikfad_checks.cuh, to *first_code);
 * *count is -1 in a library built without the checks.
 *
 * rikfad_debug_fail_allocation(n): the n-th device or page-locked host
 * allocation the library makes from now on (n >= 1, counted over all
 * threads) reports failure as if memory were exhausted; n <= 0 turns this
 * off.  It exercises the clean-up paths of rikfad_create without exhausting
 * any memory.  rikfad_debug_live_allocations returns how many allocations the
 * library currently holds (0 once every handle is destroyed).
 */
RIKFAD_API int rikfad_debug_check_failures(rikfad_handle h, int64_t *count, int *first_code);
RIKFAD_API void rikfad_debug_fail_allocation(int64_t n);
RIKFAD_API int64_t rikfad_debug_live_allocations(void);

/* Last error message of the calling thread ("" if none). */
RIKFAD_API const char *rikfad_last_error(void);

/* ABI version of this header: 1. */
RIKFAD_API int rikfad_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* RIKFAD_H */
