"""WaterKron downstream of the fit: reverse Cholesky, waterfilling scales and the
two-sided GPTQ quantizer, as a plain, slow fp64 CPU restatement.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` may import this module.  It shares no code with the CUDA library.

What it computes (paper: "WaterKron and FlipFlop Hessian", Birnick & Saab):

* Section 2, notation: RevCholesky(M) is the unique lower-triangular L with positive
  diagonal and L^T L = M.
* Section 2, Algorithm 1 (GPTQ) and Algorithm 2 (its two-sided extension): columns
  j = 1..n (and, in Algorithm 2, rows i = 1..m inside each column) are rounded in turn,
      Z_ij = round(W_ij / (alpha_j beta_i)),   V_ij = alpha_j beta_i Z_ij,
  and the error Delta = V_ij - W_ij is fed forward through the column-normalised
  inverses Lt = L^-1 (Lt[:, j] / Lt[j, j]):  W <- W + Lt^B[:, i] Delta Lt^A[:, j]^T.
* Section 3, Corollary 3.2 (waterfilling): alpha_j = sqrt(gamma) |A|^(1/2n) / L^A_jj,
  beta_i = sqrt(gamma) |B|^(1/2m) / L^B_ii.
* Section 2: two-sided distortion D_{A,B} = ||L^B (V - W) (L^A)^T||_F^2 / (m n).

Readings where the paper is silent (also listed in the design notes):
  * round() is round-to-nearest with ties to even;
  * the algorithms return Z; V = beta alpha^T (.) Z is implied by the alphabet
    (Section 2) and W itself is not returned.

All arithmetic is fp64 numpy/scipy; LAPACK's Cholesky and triangular solve are used as
library primitives.
"""
from __future__ import annotations

import numpy as np
import scipy.linalg as sla


def rev_cholesky(M: np.ndarray) -> np.ndarray:
    """Lower L with L_ii > 0 and L^T L = M (Section 2, RevCholesky).

    With the reversal permutation J (J^2 = I) and the ordinary factor C C^T = J M J
    (lower), L = J C^T J is lower triangular, has the same positive diagonal reversed,
    and L^T L = J C C^T J = M; uniqueness of the factor makes it RevCholesky(M)."""
    M = np.asarray(M, dtype=np.float64)
    C = np.linalg.cholesky(M[::-1, ::-1])
    return np.ascontiguousarray(C.T[::-1, ::-1])


def normalized_inverse(L: np.ndarray) -> np.ndarray:
    """Lt = L^-1 with every column divided by its diagonal entry (Algorithms 1 and 2,
    the normalisation step).  L lower triangular, so Lt is lower unit-triangular."""
    n = L.shape[0]
    Lt = sla.solve_triangular(L, np.eye(n), lower=True)
    return Lt / np.diag(Lt)[None, :]


def waterfilling_scales(LA: np.ndarray, LB: np.ndarray, gamma: float):
    """(alpha, beta) of Corollary 3.2: alpha_j = sqrt(gamma) |A|^(1/2n) / L^A_jj with
    |A| = prod_j (L^A_jj)^2, so |A|^(1/2n) is the geometric mean of diag(L^A)."""
    da, db = np.diag(LA), np.diag(LB)
    ga = np.exp(np.mean(np.log(da)))
    gb = np.exp(np.mean(np.log(db)))
    s = np.sqrt(gamma)
    return s * ga / da, s * gb / db


def gptq(W: np.ndarray, A: np.ndarray, alpha: np.ndarray, beta: np.ndarray) -> np.ndarray:
    """Algorithm 1 (GPTQ), step by step: returns the integer matrix Z (int64)."""
    W = np.array(W, dtype=np.float64)
    m, n = W.shape
    Lt = normalized_inverse(rev_cholesky(A))
    Z = np.zeros((m, n), dtype=np.int64)
    for j in range(n):
        z = np.rint(W[:, j] / (alpha[j] * beta))
        Z[:, j] = z
        V = alpha[j] * beta * z
        delta = V - W[:, j]
        W = W + np.outer(delta, Lt[:, j])
    return Z


def gptq2(W: np.ndarray, A: np.ndarray, B: np.ndarray, alpha: np.ndarray,
          beta: np.ndarray) -> np.ndarray:
    """Algorithm 2 (two-sided GPTQ), step by step: for j = 1..n, i = 1..m, round the
    entry and add Lt^B[:, i] Delta Lt^A[:, j]^T to W.  Returns Z (int64)."""
    LtA = normalized_inverse(rev_cholesky(A))
    LtB = normalized_inverse(rev_cholesky(B))
    return gptq2_factors(W, LtA, LtB, alpha, beta)


def gptq2_factors(W: np.ndarray, LtA: np.ndarray, LtB: np.ndarray, alpha: np.ndarray,
                  beta: np.ndarray, tie_distance: bool = False):
    """The loop of Algorithm 2 from its column-normalised inverse factors Lt^A (n x n),
    Lt^B (m x m).  Returns Z (int64), and with tie_distance also the smallest
    |frac(W_ij / (alpha_j beta_i)) - 1/2| over the decisions (how far the run stays from
    a rounding tie, so a comparison in another precision knows whether Z is unique)."""
    W = np.array(W, dtype=np.float64)
    LtA = np.asarray(LtA, dtype=np.float64)
    LtB = np.asarray(LtB, dtype=np.float64)
    alpha = np.asarray(alpha, dtype=np.float64)
    beta = np.asarray(beta, dtype=np.float64)
    m, n = W.shape
    Z = np.zeros((m, n), dtype=np.int64)
    best = np.inf
    for j in range(n):
        for i in range(m):
            t = W[i, j] / (alpha[j] * beta[i])
            if tie_distance:
                best = min(best, abs(abs(t - np.floor(t)) - 0.5))
            z = np.rint(t)
            Z[i, j] = z
            delta = alpha[j] * beta[i] * z - W[i, j]
            # Lt^B[:, i] is zero above row i and Lt^A[:, j] above row j
            W[i:, j:] += delta * np.outer(LtB[i:, i], LtA[j:, j])
    return (Z, float(best)) if tie_distance else Z


def dequantize(Z: np.ndarray, alpha: np.ndarray, beta: np.ndarray) -> np.ndarray:
    """V = beta alpha^T (.) Z (Section 2, the alphabet)."""
    return beta[:, None] * alpha[None, :] * np.asarray(Z, dtype=np.float64)


def distortion(W: np.ndarray, V: np.ndarray, A: np.ndarray, B: np.ndarray) -> float:
    """D_{A,B} = ||L^B (V - W) (L^A)^T||_F^2 / (m n) (Section 2, two-sided distortion)."""
    LA, LB = rev_cholesky(A), rev_cholesky(B)
    E = LB @ (np.asarray(V, np.float64) - np.asarray(W, np.float64)) @ LA.T
    return float(np.sum(E * E) / E.size)
