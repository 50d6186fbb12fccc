"""FlipFlop Hessian oracle: a plain, slow, fp64 CPU restatement of the estimator.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its ``cpu_baseline`` leg and ``--impl reference``) may import this
module.  It shares no code with the CUDA library and never imports it.

What it computes (paper: "WaterKron and FlipFlop Hessian", Birnick & Saab):

* H = E[x x^T (x) g g^T] for calibration pairs (x_k, g_k), G_k = g_k x_k^T,
  vec(G_k) = x_k (x) g_k (Section 5, problem statement).
* The mismatch factor Phi(H, A (x) B) (Section 4, its definition) is minimised,
  up to scale, by the alternating updates (Section 5, the flip-flop equations)
      A  propto  E[(g^T B^-1 g) x x^T]          (A-update, B fixed)
      B  propto  E[(x^T A^-1 x) g g^T]          (B-update, A fixed)
  and each half-step is the exact minimiser of its block (Section 5, the AM-GM
  argument), so the Gaussian log-likelihood (Section 4, the KL relation) never
  decreases.
* Settings of Appendix B: A_0 = I_n, one iteration = B-update then A-update;
  optional damping  F <- F + lambda * mean(diag F) * I  after each update.

Readings where the paper is silent (each also listed in the design notes):
  * "propto" is fixed by the matrix-normal MLE constants 1/(N n) for B and 1/(N m)
    for A (Dutilleul's flip-flop, cited in Section 5); afterwards tr(A) = n and
    B carries the scale (the product A (x) B is unchanged);
  * expectations are empirical means over the N samples;
  * delta_t = max over F in {A, B} of ||F^_t - F^_{t-1}||_F / ||F^_t||_F with
    F^ = F / tr F, delta_1 = +inf; the fit stops when delta_t < tol (tol = 0:
    exactly `iters` iterations);
  * quadratic forms use the lower Cholesky factor L (L L^T = F, Section 2
    notation) and forward substitution: v^T F^-1 v = ||L^-1 v||^2.

All arithmetic is fp64 numpy/scipy; LAPACK's Cholesky, triangular solve and BLAS
matmul are used as library primitives.  The only grouping of our own is that the sums
over the N samples (the empirical expectations) are accumulated over consecutive
blocks of rows, so that samples stored in a narrow type (bf16) are widened to fp64 one
block at a time and the full-size workloads fit in host memory; the sum and its terms
are unchanged, only the order of the additions.
"""
from __future__ import annotations

import dataclasses
import math
from typing import List, Optional

import numpy as np
import scipy.linalg as sla


def as_f64(a) -> np.ndarray:
    """Widen a numpy array or torch tensor (any float dtype, incl. bf16) to fp64."""
    if hasattr(a, "detach"):
        a = a.detach().to("cpu")
        import torch  # local: the oracle itself does not depend on torch

        a = a.to(torch.float64).numpy()
    return np.ascontiguousarray(np.asarray(a, dtype=np.float64))


# ----------------------------------------------------------------------------
# single steps
# ----------------------------------------------------------------------------
def cholesky(F: np.ndarray) -> np.ndarray:
    """Lower L with L L^T = F and L_ii > 0 (Section 2, Cholesky).  Raises
    numpy.linalg.LinAlgError if F is not positive definite."""
    return np.linalg.cholesky(F)


def logdet_from_cholesky(L: np.ndarray) -> float:
    """log|F| = 2 sum_i log L_ii."""
    return 2.0 * float(np.sum(np.log(np.diag(L))))


def tri_inverse(L: np.ndarray) -> np.ndarray:
    """M = L^-1 for lower-triangular L (lower-triangular), by forward substitution
    of the identity."""
    return sla.solve_triangular(L, np.eye(L.shape[0]), lower=True)


def inv_quad_forms_chol(L: np.ndarray, V: np.ndarray) -> np.ndarray:
    """q_k = v_k^T F^-1 v_k = ||L^-1 v_k||^2 for every row v_k of V (N x d), by
    forward substitution with the Cholesky factor L of F (Section 5: the weights
    x^T A^-1 x and g^T B^-1 g of the flip-flop updates)."""
    Y = sla.solve_triangular(L, V.T, lower=True)
    return np.einsum("ik,ik->k", Y, Y)


# rows widened to fp64 at a time by the fits (a block of 16384 rows of 14336 features
# is 1.9 GB)
BLOCK_ROWS = 16384


def row_blocks(V, rows: int = BLOCK_ROWS):
    """Yield (r0, r1, fp64 copy of rows r0..r1-1) of V (numpy array or torch tensor of
    any float dtype)."""
    N = V.shape[0]
    for r0 in range(0, N, rows):
        r1 = min(N, r0 + rows)
        yield r0, r1, as_f64(V[r0:r1])


def inv_quad_forms_rows(L: np.ndarray, V, rows: int = BLOCK_ROWS) -> np.ndarray:
    """inv_quad_forms_chol over all rows of V, a block of rows at a time."""
    q = np.empty(V.shape[0])
    for r0, r1, Vb in row_blocks(V, rows):
        q[r0:r1] = inv_quad_forms_chol(L, Vb)
    return q


def sq_norms_rows(V, rows: int = BLOCK_ROWS) -> np.ndarray:
    """||v_k||^2 = v_k^T I^-1 v_k for every row (the weights at A_0 = I)."""
    q = np.empty(V.shape[0])
    for r0, r1, Vb in row_blocks(V, rows):
        q[r0:r1] = np.einsum("kd,kd->k", Vb, Vb)
    return q


def weighted_gram_rows(V, w: np.ndarray, scale: float, rows: int = BLOCK_ROWS) -> np.ndarray:
    """scale * sum_k w_k v_k v_k^T (weighted_gram), the sum over k accumulated a block
    of rows at a time."""
    d = V.shape[1]
    C = np.zeros((d, d))
    for r0, r1, Vb in row_blocks(V, rows):
        C += weighted_gram(Vb, w[r0:r1], 1.0)
    return scale * C


def fwd_quad_forms(F: np.ndarray, V: np.ndarray) -> np.ndarray:
    """q_k = v_k^T F v_k (the Frobenius variant's weights, Section 5)."""
    return np.einsum("kd,kd->k", V @ F, V)


def weighted_gram(V: np.ndarray, w: np.ndarray, scale: float) -> np.ndarray:
    """scale * sum_k w_k v_k v_k^T = scale * V^T diag(w) V (Section 5: the
    expectations E[(.) x x^T] and E[(.) g g^T] as empirical means).  With all w_k >= 0
    (the flip-flop weights are quadratic forms of SPD matrices) each term is written
    (sqrt(w_k) v_k)(sqrt(w_k) v_k)^T, so the product is a symmetric rank-k update."""
    w = np.asarray(w, dtype=np.float64)
    if np.all(w >= 0.0):
        Vs = V * np.sqrt(w)[:, None]
        return scale * (Vs.T @ Vs)
    return scale * ((V.T * w) @ V)


def damp(F: np.ndarray, lam: float) -> np.ndarray:
    """F + lam * mean(diag F) * I (Appendix B damping; mean taken before the shift)."""
    if lam == 0.0:
        return F
    return F + lam * float(np.mean(np.diag(F))) * np.eye(F.shape[0])


def gaussian_loglik(N: int, n: int, m: int, logdet_A: float, logdet_B: float,
                    sum_trace: float) -> float:
    """Matrix-normal log-likelihood of the N samples vec(G_k) ~ N(0, A (x) B) up to
    the constant -N m n log(2 pi)/2:  -1/2 [N m log|A| + N n log|B| + sum_k
    tr(B^-1 G_k A^-1 G_k^T)]; for G_k = g_k x_k^T the trace is q_k r_k (Section 5
    trace identity, Section 4 KL relation)."""
    return -0.5 * (N * m * logdet_A + N * n * logdet_B + sum_trace)


def loglik(X, G, A, B) -> float:
    """Evaluate the rank-one log-likelihood from scratch at (A, B)."""
    X, G, A, B = as_f64(X), as_f64(G), as_f64(A), as_f64(B)
    N, n = X.shape
    m = G.shape[1]
    LA, LB = cholesky(A), cholesky(B)
    q = inv_quad_forms_chol(LA, X)
    r = inv_quad_forms_chol(LB, G)
    return gaussian_loglik(N, n, m, logdet_from_cholesky(LA), logdet_from_cholesky(LB),
                           float(np.dot(q, r)))


def phi_tilde(X, G, A, B) -> float:
    """Scale-free mismatch factor for empirical (possibly singular) H:
    Phi~ = |A|^{1/n} |B|^{1/m} * tr(H (A (x) B)^-1) / (m n), with
    tr(H (A (x) B)^-1) = mean_k q_k r_k (Section 5), i.e. Phi times |H|^{1/mn}."""
    X, G, A, B = as_f64(X), as_f64(G), as_f64(A), as_f64(B)
    n, m = X.shape[1], G.shape[1]
    LA, LB = cholesky(A), cholesky(B)
    q = inv_quad_forms_chol(LA, X)
    r = inv_quad_forms_chol(LB, G)
    log_phi = (logdet_from_cholesky(LA) / n + logdet_from_cholesky(LB) / m
               + math.log(float(np.mean(q * r)) / (m * n)))
    return math.exp(log_phi)


def normalized(F: np.ndarray) -> np.ndarray:
    return F / np.trace(F)


def rel_change(F_new: np.ndarray, F_old: np.ndarray) -> float:
    a, b = normalized(F_new), normalized(F_old)
    return float(np.linalg.norm(a - b) / np.linalg.norm(a))


# ----------------------------------------------------------------------------
# the fit
# ----------------------------------------------------------------------------
@dataclasses.dataclass
class FitResult:
    A: np.ndarray
    B: np.ndarray
    iters_done: int
    deltas: List[float]
    # log-likelihood after each half-step: [l(A_0,B_1), l(A_1,B_1), l(A_1,B_2), ...]
    loglik: List[float]
    # mean_k q_k r_k after each half-step (the trace identity gives m n)
    mean_qr: List[float]
    q: Optional[np.ndarray] = None   # last q (x^T A^-1 x with the returned A)
    r: Optional[np.ndarray] = None   # last r (g^T B^-1 g with the returned B)
    # (A_t, B_t) after every iteration, when asked for
    iterates: List = dataclasses.field(default_factory=list)


def flipflop_fit(X, G, iters: int, tol: float = 0.0, damping: float = 0.0,
                 init_A=None, rows: int = BLOCK_ROWS, keep_iterates: bool = False,
                 progress=None) -> FitResult:
    """FlipFlop Hessian fit of A (n x n) and B (m x m) to rank-one samples.

    X: N x n (rows x_k^T), G: N x m (rows g_k^T), numpy arrays or host torch tensors
    of any float dtype (widened to fp64 a block of `rows` rows at a time).  Section 5
    flip-flop updates with the Appendix B settings (A_0 = I_n unless init_A is given;
    iteration = B-update, then A-update), MLE constants, tr(A) = n normalisation after
    each iteration.  keep_iterates: also return every (A_t, B_t).  progress: called
    with (t, delta_t) after each iteration.
    """
    if not hasattr(X, "shape") or not hasattr(G, "shape"):
        X, G = as_f64(X), as_f64(G)
    N, n = X.shape
    m = G.shape[1]
    if init_A is None:
        A = np.eye(n)
        q = sq_norms_rows(X, rows)                # x^T I^-1 x
        logdet_A = 0.0
    else:
        A = as_f64(init_A)
        LA = cholesky(A)
        q = inv_quad_forms_rows(LA, X, rows)
        logdet_A = logdet_from_cholesky(LA)
    B_prev = None
    A_prev = A.copy()
    deltas, lls, mqr = [], [], []
    iterates = []
    t_done = 0
    r = None
    for t in range(1, iters + 1):
        # B-update with A fixed: B = 1/(N n) sum_k q_k g_k g_k^T
        B = damp(weighted_gram_rows(G, q, 1.0 / (N * n), rows), damping)
        LB = cholesky(B)
        logdet_B = logdet_from_cholesky(LB)
        r = inv_quad_forms_rows(LB, G, rows)
        lls.append(gaussian_loglik(N, n, m, logdet_A, logdet_B, float(np.dot(q, r))))
        mqr.append(float(np.mean(q * r)))
        # A-update with B fixed: A = 1/(N m) sum_k r_k x_k x_k^T
        A = damp(weighted_gram_rows(X, r, 1.0 / (N * m), rows), damping)
        # scale freedom: tr(A) = n, B carries the scale
        s = np.trace(A) / n
        A = A / s
        B = B * s
        logdet_B += m * math.log(s)
        r = r / s
        LA = cholesky(A)
        logdet_A = logdet_from_cholesky(LA)
        q = inv_quad_forms_rows(LA, X, rows)
        lls.append(gaussian_loglik(N, n, m, logdet_A, logdet_B, float(np.dot(q, r))))
        mqr.append(float(np.mean(q * r)))
        delta = math.inf if B_prev is None else max(rel_change(A, A_prev),
                                                    rel_change(B, B_prev))
        deltas.append(delta)
        A_prev, B_prev = A.copy(), B.copy()
        if keep_iterates:
            iterates.append((A_prev, B_prev))
        t_done = t
        if progress is not None:
            progress(t, delta)
        if tol > 0.0 and delta < tol:
            break
    return FitResult(A=A, B=B, iters_done=t_done, deltas=deltas, loglik=lls,
                     mean_qr=mqr, q=q, r=r, iterates=iterates)


def flipflop_fit_matrix(Gk, iters: int, tol: float = 0.0, damping: float = 0.0,
                        init_A=None) -> FitResult:
    """FlipFlop fit to general matrix samples G_k in R^{m x n} (N x m x n):
        B = 1/(N n) sum_k G_k A^-1 G_k^T,   A = 1/(N m) sum_k G_k^T B^-1 G_k
    (Section 5, the first form of each update), i.e. the matrix-normal MLE
    flip-flop.  Same order, constants and normalisation as flipflop_fit."""
    Gk = as_f64(Gk)
    N, m, n = Gk.shape
    A = np.eye(n) if init_A is None else as_f64(init_A)
    # columns of the stacked matrices: (G_k^T)[:, i] for all k, i  and  G_k[:, j]
    GT_stack = Gk.transpose(2, 0, 1).reshape(n, N * m)
    G_stack = Gk.transpose(1, 0, 2).reshape(m, N * n)
    LA = cholesky(A)
    logdet_A = logdet_from_cholesky(LA)
    B_prev, A_prev = None, A.copy()
    deltas, lls, mqr = [], [], []
    t_done = 0
    B = None
    for t in range(1, iters + 1):
        # W_k = L_A^-1 G_k^T (n x m); G_k A^-1 G_k^T = W_k^T W_k
        W = sla.solve_triangular(LA, GT_stack, lower=True).reshape(n, N, m)
        B = damp(np.einsum("jki,jkl->il", W, W) / (N * n), damping)
        LB = cholesky(B)
        logdet_B = logdet_from_cholesky(LB)
        # Y_k = L_B^-1 G_k (m x n); G_k^T B^-1 G_k = Y_k^T Y_k
        Y = sla.solve_triangular(LB, G_stack, lower=True).reshape(m, N, n)
        # tr(B^-1 G_k A^-1 G_k^T) = ||L_B^-1 G_k L_A^-T||_F^2
        tr_sum = _sum_sq_two_sided(Y, LA)
        lls.append(gaussian_loglik(N, n, m, logdet_A, logdet_B, tr_sum))
        mqr.append(tr_sum / N)
        A = damp(np.einsum("ikj,ikl->jl", Y, Y) / (N * m), damping)
        s = np.trace(A) / n
        A, B = A / s, B * s
        logdet_B += m * math.log(s)
        LA = cholesky(A)
        logdet_A = logdet_from_cholesky(LA)
        LB = cholesky(B)
        Y = sla.solve_triangular(LB, G_stack, lower=True).reshape(m, N, n)
        tr_sum = _sum_sq_two_sided(Y, LA)
        lls.append(gaussian_loglik(N, n, m, logdet_A, logdet_B, tr_sum))
        mqr.append(tr_sum / N)
        delta = math.inf if B_prev is None else max(rel_change(A, A_prev),
                                                    rel_change(B, B_prev))
        deltas.append(delta)
        A_prev, B_prev = A.copy(), B.copy()
        t_done = t
        if tol > 0.0 and delta < tol:
            break
    return FitResult(A=A, B=B, iters_done=t_done, deltas=deltas, loglik=lls, mean_qr=mqr)


def flipflop_fit_matrix_blocks(sample_blocks, N: int, m: int, n: int, iters: int,
                               tol: float = 0.0, damping: float = 0.0, progress=None):
    """flipflop_fit_matrix for samples too large to hold at once: sample_blocks() yields
    consecutive blocks G_k (b x m x n, any float dtype) covering all N samples, and may
    be called once per half-step.  Same updates, constants, order and normalisation; each
    expectation is accumulated block by block.  Returns (A, B, iters_done, deltas); the
    log-likelihood statistics are not evaluated."""
    A = np.eye(n)
    B_prev, A_prev = None, A.copy()
    deltas = []
    t_done = 0
    B = None
    for t in range(1, iters + 1):
        LA = cholesky(A)
        # B = 1/(N n) sum_k G_k A^-1 G_k^T = sum_k W_k^T W_k with W_k = L_A^-1 G_k^T
        acc = np.zeros((m, m))
        for Gb in sample_blocks():
            Gb = as_f64(Gb)
            b = Gb.shape[0]
            W = sla.solve_triangular(LA, Gb.transpose(2, 0, 1).reshape(n, b * m), lower=True)
            W = W.reshape(n, b, m).transpose(1, 0, 2).reshape(b * n, m)   # rows (k, i)
            acc += W.T @ W
        B = damp(acc / (N * n), damping)
        LB = cholesky(B)
        # A = 1/(N m) sum_k G_k^T B^-1 G_k = sum_k Y_k^T Y_k with Y_k = L_B^-1 G_k
        acc = np.zeros((n, n))
        for Gb in sample_blocks():
            Gb = as_f64(Gb)
            b = Gb.shape[0]
            Y = sla.solve_triangular(LB, Gb.transpose(1, 0, 2).reshape(m, b * n), lower=True)
            Y = Y.reshape(m, b, n).transpose(1, 0, 2).reshape(b * m, n)   # rows (k, j)
            acc += Y.T @ Y
        A = damp(acc / (N * m), damping)
        s = np.trace(A) / n
        A, B = A / s, B * s
        delta = math.inf if B_prev is None else max(rel_change(A, A_prev),
                                                    rel_change(B, B_prev))
        deltas.append(delta)
        A_prev, B_prev = A.copy(), B.copy()
        t_done = t
        if progress is not None:
            progress(t, delta)
        if tol > 0.0 and delta < tol:
            break
    return A, B, t_done, deltas


def _sum_sq_two_sided(Y: np.ndarray, LA: np.ndarray) -> float:
    """sum_k ||Y_k L_A^-T||_F^2 for Y of shape (m, N, n)."""
    m, N, n = Y.shape
    Z = sla.solve_triangular(LA, Y.transpose(2, 0, 1).reshape(n, m * N), lower=True)
    return float(np.sum(Z * Z))


# ----------------------------------------------------------------------------
# the comparison Hessians of Table 1
# ----------------------------------------------------------------------------
def input_hessian(X, m: int):
    """Table 1 "Input": A = E[x x^T], B = I_m."""
    X = as_f64(X)
    return X.T @ X / X.shape[0], np.eye(m)


def marginal_hessian(X, G):
    """Table 1 "Marginal": A = E[x x^T], B = E[g g^T]."""
    X, G = as_f64(X), as_f64(G)
    N = X.shape[0]
    return X.T @ X / N, G.T @ G / N


def frobenius_fit(X, G, iters: int) -> FitResult:
    """Table 1 "Frobenius": the flip-flop loop with A^-1, B^-1 replaced by A, B
    (Section 5, last paragraph), i.e. alternating least squares for
    min ||H - A (x) B||_F:  B = E[(x^T A x) g g^T] / ||A||_F^2,
    A = E[(g^T B g) x x^T] / ||B||_F^2.  A_0 = I_n, B-update first, tr(A) = n."""
    X, G = as_f64(X), as_f64(G)
    N, n = X.shape
    A = np.eye(n)
    B = None
    for _ in range(iters):
        q = fwd_quad_forms(A, X)
        B = weighted_gram(G, q, 1.0 / N) / float(np.sum(A * A))
        r = fwd_quad_forms(B, G)
        A = weighted_gram(X, r, 1.0 / N) / float(np.sum(B * B))
        s = np.trace(A) / n
        A, B = A / s, B * s
    return FitResult(A=A, B=B, iters_done=iters, deltas=[], loglik=[], mean_qr=[])


# ----------------------------------------------------------------------------
# parity metric
# ----------------------------------------------------------------------------
def kron_rel_err(A, B, A_ref, B_ref) -> float:
    """||A^ (x) B^ - A^' (x) B^'||_F / ||A^' (x) B^'||_F with F^ = F / tr F, in
    closed form (||P (x) Q||_F = ||P||_F ||Q||_F, <P (x) Q, P' (x) Q'> =
    <P,P'><Q,Q'>), without forming the mn x mn products.  The fixed point is
    unique only up to the scale (cA, B/c) (Section 5), so the metric is
    scale-free."""
    a, b = normalized(as_f64(A)), normalized(as_f64(B))
    a2, b2 = normalized(as_f64(A_ref)), normalized(as_f64(B_ref))
    num2 = (np.sum(a * a) * np.sum(b * b) + np.sum(a2 * a2) * np.sum(b2 * b2)
            - 2.0 * np.sum(a * a2) * np.sum(b * b2))
    den2 = np.sum(a2 * a2) * np.sum(b2 * b2)
    return float(math.sqrt(max(num2, 0.0) / den2))


def factor_rel_errs(A, B, A_ref, B_ref):
    """(||A^ - A^'||_F / ||A^'||_F, same for B): stays accurate below ~1e-8, where
    the closed-form Kronecker metric cancels."""
    a, b = normalized(as_f64(A)), normalized(as_f64(B))
    a2, b2 = normalized(as_f64(A_ref)), normalized(as_f64(B_ref))
    return (float(np.linalg.norm(a - a2) / np.linalg.norm(a2)),
            float(np.linalg.norm(b - b2) / np.linalg.norm(b2)))
