/*
 * ffh.h -- C ABI of libffh, the FlipFlop Hessian estimator on one GB300 GPU.
 *
 * The estimator (Birnick & Saab, "WaterKron and FlipFlop Hessian", Section 5) fits a
 * Kronecker-factored Hessian A (x) B, A in R^{n x n} (input side), B in R^{m x m}
 * (output side), to the calibration samples of a linear layer W in R^{m x n}.  For
 * rank-one samples G_k = g_k x_k^T (x_k in R^n the layer input, g_k in R^m the output
 * gradient) the flip-flop updates are
 *
 *     B <- 1/(N n) sum_k (x_k^T A^-1 x_k) g_k g_k^T,
 *     A <- 1/(N m) sum_k (g_k^T B^-1 g_k) x_k x_k^T,
 *
 * iterated from A_0 = I_n, one iteration = B-update then A-update (Appendix B).  The
 * proportionality constants of Section 5 are fixed to the matrix-normal MLE values
 * above; after every iteration A is rescaled to tr(A) = n and B by the inverse
 * factor, which leaves A (x) B unchanged (the fixed point is unique only up to that
 * scale).
 *
 * Conventions common to every call:
 *  - Matrices are row-major.  X is N x n (row k = x_k^T), G is N x m (row k = g_k^T),
 *    Gk is N x m x n (sample k is the m x n matrix G_k).  A is n x n, B is m x m, both
 *    written in full symmetric storage, fp32.
 *  - "device or host": a pointer may address device memory or host memory (pinned or
 *    pageable).  Host inputs are copied into the handle's workspace and host outputs
 *    copied back inside the call; device inputs are read in place.  All device memory
 *    passed in is owned by the caller and must stay valid until the call returns.
 *  - Every call enqueues its work on the handle's CUDA stream and synchronises that
 *    stream once before returning (the status of the fit is read back then).
 *  - A handle must not be used by two host threads at once.  Each handle owns a
 *    workspace on the current device, grown on demand and freed by ffh_destroy.
 *  - On error the outputs are undefined; ffh_last_error() describes the error.
 */
#ifndef FFH_H
#define FFH_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct ffh_ctx* ffh_t;

typedef enum {
  FFH_OK = 0,
  FFH_ERR_INVALID_ARG = 1, /* null pointer, bad size, misaligned row pitch, iters < 1 */
  FFH_ERR_NOT_SPD = 2,     /* a Cholesky pivot was <= 0 or not finite */
  FFH_ERR_RANK = 3,        /* N < max(n, m) without damping: the MLE need not exist */
  FFH_ERR_OOM = 4,         /* workspace allocation failed */
  FFH_ERR_CUDA = 5,        /* a CUDA runtime call failed */
  FFH_ERR_TIMEOUT = 6,     /* a bounded device-side wait expired; the kernel returned */
  FFH_ERR_UNSUPPORTED = 7  /* no sm_100-family GPU, or an option this library version lacks */
} ffh_status;

typedef enum { FFH_BF16 = 0, FFH_F32 = 1 } ffh_dtype;

/* The Hessian approximations of Table 1 (all returned with tr(A) = n, B carrying the
 * scale; only the product A (x) B is defined by the paper). */
typedef enum {
  FFH_FLIPFLOP = 0,  /* A = E[(g^T B^-1 g) x x^T], B = E[(x^T A^-1 x) g g^T] (Section 5) */
  FFH_FROBENIUS = 1, /* A = E[(g^T B g) x x^T]/||B||_F^2, B = E[(x^T A x) g g^T]/||A||_F^2:
                        alternating least squares for min ||H - A (x) B||_F (Section 5,
                        last paragraph); same A_0 = I and B-then-A order */
  FFH_INPUT = 2,     /* A = E[x x^T], B = I_m (one pass; iters ignored) */
  FFH_MARGINAL = 3   /* A = E[x x^T], B = E[g g^T] (one pass; iters ignored) */
} ffh_variant;

/* Test-only fault injection codes (ffh_options.fault). */
enum {
  FFH_FAULT_NONE = 0,
  FFH_FAULT_OOM = 1,          /* the next workspace allocation reports failure */
  FFH_FAULT_BAD_PIVOT = 2,    /* the first Cholesky sees a NaN pivot -> FFH_ERR_NOT_SPD */
  FFH_FAULT_LOST_COPY = 3     /* the Gram kernel drops one staged copy, so its consumer's
                                 bounded wait expires -> FFH_ERR_TIMEOUT (device context
                                 stays usable) */
};

/* Zero-initialised options are the defaults. */
typedef struct {
  int32_t dtype;           /* ffh_dtype of X and G (Gk is always fp32) */
  float damping;           /* lambda >= 0: F <- F + lambda * mean(diag F) * I right after
                              each update, the mean taken before the shift (Appendix B
                              uses 0.1; default 0) */
  int32_t variant;         /* ffh_variant */
  const float* init_A;     /* optional warm start (n x n fp32, SPD, device or host);
                              NULL: A_0 = I_n (Appendix B) */
  int32_t final_loglik;    /* 1: also evaluate the log-likelihood at the returned (A, B)
                              (one more Cholesky and quadratic-form pass) */
  int32_t reserved0;       /* must be zero */
  int32_t fault;           /* FFH_FAULT_* (tests only) */
  int32_t profile;         /* 1: time the Gram, quadratic-form and Cholesky kernels with
                              CUDA events on the handle's stream (see ffh_get_timings) */
  int32_t no_graph;        /* 0 (default): ffh_fit with device-resident X and G records the
                              work it enqueues as a CUDA graph the first time and replays it
                              when the next fit on the handle has the same sizes, pointers,
                              iters, tol and options (one launch instead of thousands);
                              1: always enqueue kernel by kernel */
  int32_t reserved[3];     /* must be zero */
} ffh_options;

/* Kernel timings accumulated over the calls made with opt.profile = 1. */
typedef struct {
  double gram_ms;          /* total device time of the weighted-Gram main kernel */
  int64_t gram_launches;
  double qform_ms;         /* total device time of the quadratic-form kernel */
  int64_t qform_launches;
  double chol_ms;          /* total device time of Cholesky + inverse (all their kernels) */
  int64_t chol_calls;
  int64_t kernel_launches; /* every kernel libffh launched in this process (profile or not) */
} ffh_timings;

/* Library version as major*10000 + minor*100 + patch. */
int32_t ffh_version(void);

/* Create a handle bound to the current CUDA device and to `cuda_stream` (a
 * cudaStream_t; NULL = the legacy default stream).  `opt` may be NULL (defaults).
 * Fails with FFH_ERR_UNSUPPORTED unless the device is compute capability 10.x. */
ffh_status ffh_create(ffh_t* out, const ffh_options* opt, void* cuda_stream);

/* Replace the options / the stream of an existing handle. */
ffh_status ffh_set_options(ffh_t h, const ffh_options* opt);
ffh_status ffh_set_stream(ffh_t h, void* cuda_stream);

/* Free the workspace and the handle.  NULL is accepted. */
ffh_status ffh_destroy(ffh_t h);

/* Human-readable description of the last error on this handle ("" if none).  The
 * string is owned by the handle and valid until its next call. */
const char* ffh_last_error(ffh_t h);

/* FlipFlop fit to rank-one samples (Section 5 updates, Appendix B settings).
 *   X      N x n, row pitch n elements, dtype opt.dtype (device or host)
 *   G      N x m, row pitch m elements, same dtype
 *   iters  maximum number of iterations (>= 1); one iteration = B-update, A-update
 *   tol    stop after iteration t when delta_t < tol, where
 *          delta_t = max_{F in {A,B}} ||F_t/tr F_t - F_{t-1}/tr F_{t-1}||_F / ||F_t/tr F_t||_F
 *          (delta_1 = +inf); tol = 0 runs exactly `iters` iterations.  The test runs on
 *          the device: all `iters` iterations are enqueued, those after the stop return
 *          at once, and the host synchronises once per call, at the end
 *   A_out  n x n fp32 (device or host): A with tr(A) = n
 *   B_out  m x m fp32 (device or host)
 * bf16 rows must be 16-byte aligned: n and m multiples of 8 for FFH_BF16 (fp32 inputs
 * accept any n, m).  Reaching `iters` without meeting `tol` is not an error; see
 * ffh_get_stats.  Errors: INVALID_ARG, RANK, NOT_SPD, OOM, CUDA, TIMEOUT. */
ffh_status ffh_fit(ffh_t h, const void* X, const void* G, int64_t N, int64_t n, int64_t m,
                   int32_t iters, float tol, float* A_out, float* B_out);

/* FlipFlop fit to general matrix samples G_k in R^{m x n} (Section 5, the first form of
 * each update):  B <- 1/(N n) sum_k G_k A^-1 G_k^T,  A <- 1/(N m) sum_k G_k^T B^-1 G_k.
 *   Gk  N x m x n fp32, row-major per sample (device or host).
 * Other arguments, normalisation and errors as ffh_fit.  n and m multiples of 4. */
ffh_status ffh_fit_matrix(ffh_t h, const float* Gk, int64_t N, int64_t n, int64_t m,
                          int32_t iters, float tol, float* A_out, float* B_out);

/* Statistics of the last fit on this handle (host pointers, each nullable).
 *   iters_done    iterations run
 *   delta         delta of the last iteration (+inf after one iteration)
 *   loglik_trace  receives up to `capacity` values: the Gaussian log-likelihood
 *                 -1/2 [N m log|A| + N n log|B| + sum_k tr(B^-1 G_k A^-1 G_k^T)]
 *                 after every half-step: l(A_0,B_1), l(A_1,B_1), l(A_1,B_2), ...;
 *                 the last entry is NaN unless opt.final_loglik was set
 *   mean_qr       receives up to `capacity` values of mean_k q_k r_k after every
 *                 half-step (m n for an undamped fit: the trace identity)
 * Returns the number of trace entries available (2 * iters_done) via *n_trace. */
ffh_status ffh_get_stats(ffh_t h, int32_t* iters_done, double* delta, double* loglik_trace,
                         double* mean_qr, int32_t capacity, int32_t* n_trace);

/* Copy the accumulated timings into *out; reset = 1 clears them afterwards (the
 * process-wide launch counter is not reset). */
ffh_status ffh_get_timings(ffh_t h, ffh_timings* out, int32_t reset);

/* Scale-free mismatch factor of a Kronecker approximation (Section 4, its definition,
 * in the sample form of Section 5):
 *   Phi~(A, B) = |A|^{1/n} |B|^{1/m} (1/(N m n)) sum_k (x_k^T A^-1 x_k)(g_k^T B^-1 g_k)
 * which is Phi(H, A (x) B) times |H|^{1/mn} (H need not be invertible).  Smaller is
 * better; the FlipFlop fit minimises it.
 *   X, G: samples as for ffh_fit (device), A (n x n), B (m x m): fp32 SPD (device)
 *   phi_out: host double.  Errors: INVALID_ARG, NOT_SPD, CUDA. */
ffh_status ffh_phi_tilde(ffh_t h, const void* X, const void* G, int64_t N, int64_t n, int64_t m,
                         const float* A, const float* B, double* phi_out);

/* ---- single steps of the fit (device pointers only; on the handle's stream) ---- */

/* Weighted Gram (the E[w v v^T] of the Section 5 updates; w = NULL gives the plain
 * Gram E[v v^T] of Table 1's Input / Marginal Hessians):
 *   C = scale * sum_k w_k v_k v_k^T = scale * V^T diag(w) V
 *   V      N x d, row pitch d, dtype opt.dtype (bf16: d multiple of 8)
 *   w      N fp32 weights, or NULL for w = 1
 *   C_out  d x d fp32, full symmetric storage (lower triangle computed, mirrored). */
ffh_status ffh_weighted_gram(ffh_t h, const void* V, const float* w, int64_t N, int64_t d,
                             float scale, float* C_out);

/* Quadratic forms with an inverse Cholesky factor (the weights x^T A^-1 x of Section 5):
 *   q_k = ||Linv v_k||^2 = v_k^T F^-1 v_k  when Linv = L^-1, L L^T = F
 *   V      N x d (dtype opt.dtype), Linv d x d fp32 lower-triangular, q_out N fp32. */
ffh_status ffh_quad_form(ffh_t h, const void* V, const float* Linv, int64_t N, int64_t d,
                         float* q_out);

/* Cholesky factor and its inverse (Section 2 notation: L lower, L L^T = F, L_ii > 0):
 *   F        d x d fp32 symmetric (lower triangle read)
 *   L_out    d x d fp32, lower triangle (upper set to 0); nullable
 *   Linv_out d x d fp32, L^-1 (lower, upper 0); nullable
 *   logdet   host double, log|F| = 2 sum_i log L_ii; nullable
 * Errors: NOT_SPD if a pivot is <= 0 or not finite. */
ffh_status ffh_cholesky(ffh_t h, const float* F, int64_t d, float* L_out, float* Linv_out,
                        double* logdet);

/* ---- sample-sharded fit (device pointers; handle's stream) ----
 * Every update of Section 5 is an expectation, i.e. a sum over the N samples, so ranks
 * that hold disjoint shards of the samples can each form the unscaled partial sum of
 * their shard, add the partial sums over all ranks (the caller's all-reduce, e.g. NCCL),
 * and finish the update identically on every rank.  One half-step (the B-update shown;
 * the A-update swaps the roles of X and G):
 *   ffh_partial_gram(h, X_r, G_r, N_r, n, m, A, P)   on each rank r
 *   all-reduce P (sum over ranks)
 *   ffh_update_from_sum(h, P, m, 1 / (N n), B)       N = sum_r N_r
 * then ffh_normalize_pair after the A-update and ffh_relative_change for the stop test.
 * The Python driver fit_sharded (package paper_2609_14706_gb300.sharded) composes them. */

/* P = sum_k w_k v_k v_k^T over the N rows of this shard, unscaled, with
 * w_k = u_k^T F^-1 u_k (F = NULL: w_k = ||u_k||^2, i.e. F = I, the first B-update):
 *   U          N x du samples whose quadratic forms weight the sum (X for the B-update)
 *   V          N x dv samples of the Gram (G for the B-update); U, V dtype opt.dtype
 *   F          du x du fp32 SPD, or NULL
 *   accumulate 0: P_out = P;  1: P_out += P (a process holding several shards)
 *   P_out      dv x dv fp32, full symmetric
 *   logdet_F   host double, log|F| (0 for F = NULL); nullable
 * Errors: INVALID_ARG, NOT_SPD, OOM, CUDA, TIMEOUT. */
ffh_status ffh_partial_gram(ffh_t h, const void* U, const void* V, int64_t N, int64_t du,
                            int64_t dv, const float* F, int32_t accumulate, float* P_out,
                            double* logdet_F);

/* F_out = scale * P, then the handle's damping F += lambda mean(diag F) I (Appendix B):
 * the update from the partial sums added over all ranks (scale = 1/(N d_other)).
 * P, F_out: d x d fp32 (may alias).  Errors: INVALID_ARG, CUDA. */
ffh_status ffh_update_from_sum(ffh_t h, const float* P, int64_t d, double scale, float* F_out);

/* s = tr(A)/n; A <- A / s; B <- B * s (the scale freedom of Section 5); s_out nullable. */
ffh_status ffh_normalize_pair(ffh_t h, float* A, int64_t n, float* B, int64_t m, double* s_out);

/* delta = ||F/tr F - Fprev/tr Fprev||_F / ||F/tr F||_F (the fit's stopping statistic for
 * one factor); delta_out: host double. */
ffh_status ffh_relative_change(ffh_t h, const float* F, const float* Fprev, int64_t d,
                               double* delta_out);

/* ---- WaterKron downstream of the fit (Sections 2-3; device pointers, handle's stream) ---- */

/* Reverse Cholesky (Section 2 notation: RevCholesky(F) is the lower L with L_ii > 0 and
 * L^T L = F) and the column-normalised inverse used by Algorithms 1-2
 * (Lt = L^-1 with Lt[:, j] divided by Lt[j][j], so Lt is lower unit-triangular):
 *   F       d x d fp32 SPD, row-major (read only)
 *   L_out   d x d fp32 lower (zeros above); nullable
 *   Lt_out  d x d fp32 lower unit-triangular; nullable
 *   logdet  host double, log|F|; nullable
 * Computed as J C^T J from the Cholesky factor C of J F J (J the reversal).
 * Errors: NOT_SPD, INVALID_ARG, OOM, CUDA. */
ffh_status ffh_rev_cholesky(ffh_t h, const float* F, int64_t d, float* L_out, float* Lt_out,
                            double* logdet);

/* Waterfilling scales of Corollary 3.2 (Section 3):
 *   alpha_j = sqrt(gamma) |A|^(1/2n) / L^A_jj,   beta_i = sqrt(gamma) |B|^(1/2m) / L^B_ii
 *   LA n x n = RevCholesky(A), LB m x m = RevCholesky(B) (ffh_rev_cholesky); only the
 *   diagonals are read.  alpha_out n fp32, beta_out m fp32; gamma > 0 sets the rate. */
ffh_status ffh_waterfilling_scales(ffh_t h, const float* LA, int64_t n, const float* LB, int64_t m,
                                   float gamma, float* alpha_out, float* beta_out);

/* Two-sided GPTQ quantizer (Algorithm 2): for j = 0..n-1, i = 0..m-1,
 *   Z_ij = round(W_ij / (alpha_j beta_i)) (nearest, ties to even),
 *   W <- W + Lt^B[:, i] (alpha_j beta_i Z_ij - W_ij) Lt^A[:, j]^T
 *   W      m x n fp32, row-major (read only; the feedback goes to a library copy)
 *   LtA    n x n, LtB m x m: column-normalised inverses from ffh_rev_cholesky
 *   alpha  n fp32 > 0, beta m fp32 > 0 (e.g. ffh_waterfilling_scales)
 *   Z_out  m x n int32; V_out m x n fp32 = beta alpha^T (.) Z, nullable
 * m <= 32768 (one column of feedback per CTA in shared memory).
 * Errors: INVALID_ARG, OOM, TIMEOUT (a bounded wait between columns expired), CUDA. */
ffh_status ffh_gptq2(ffh_t h, const float* W, const float* LtA, const float* LtB,
                     const float* alpha, const float* beta, int64_t m, int64_t n, int32_t* Z_out,
                     float* V_out);

/* Weighted Gram that allocates no device memory.  The paper has no counterpart: this
 * entry point exists for callers that cannot call cudaMalloc -- code running inside a
 * framework that owns all device memory (a pre-reserved pool, an inference-engine
 * plugin) or a latency-critical path where an allocation would synchronise the device.
 *   Computes the same C = scale * V^T diag(w) V as ffh_weighted_gram (bf16 V, N x d,
 *   d a multiple of 8; w N fp32 or NULL; C_out d x d fp32), with no handle.
 *   V, w, C_out: device pointers owned by the caller.  cuda_stream: cudaStream_t.
 *   errbuf / errbuf_len: optional caller buffer that receives a message.
 * Working memory comes from one static device array of 64 MiB that the library holds
 * on every GPU where it is loaded, until the process exits; N, d whose working memory
 * does not fit (roughly d > 5000) are rejected with FFH_ERR_INVALID_ARG before any
 * GPU work.  The first call on a device looks up the array's address (set-up); make
 * that first call before any stream capture.  All calls share the array and it keeps
 * the last call's contents (this call clears what must start at zero): calls whose
 * work overlaps on the GPU race and must be serialised by the caller.  The call
 * synchronises `cuda_stream` once to read the status word. */
ffh_status ffh_weighted_gram_static(const void* V, const float* w, int64_t N, int64_t d,
                                    float scale, float* C_out, void* cuda_stream,
                                    char* errbuf, int32_t errbuf_len);

#ifdef __cplusplus
}
#endif
#endif /* FFH_H */
