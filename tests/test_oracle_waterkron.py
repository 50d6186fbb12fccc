"""Pins of the WaterKron oracle (reverse Cholesky, waterfilling scales, two-sided GPTQ)
against what the paper and the mathematics fix, independent of the oracle's own code."""
import math

import numpy as np
import pytest

from oracle import waterkron as wk


def _spd(n, seed, cond=30.0):
    rng = np.random.default_rng(seed)
    Q, _ = np.linalg.qr(rng.standard_normal((n, n)))
    lam = np.geomspace(1.0, cond, n)
    return (Q * lam) @ Q.T


def test_rev_cholesky_worked_example():
    """Section 3, Figure 1: L = [[2, 0], [1, 3]] is RevCholesky of L^T L."""
    L = np.array([[2.0, 0.0], [1.0, 3.0]])
    assert np.allclose(wk.rev_cholesky(L.T @ L), L, atol=1e-14)


def test_rev_cholesky_definition():
    """Lower triangular, positive diagonal, L^T L = M (Section 2 notation)."""
    M = _spd(40, 1)
    L = wk.rev_cholesky(M)
    assert np.allclose(np.triu(L, 1), 0.0)
    assert np.all(np.diag(L) > 0)
    assert np.allclose(L.T @ L, M, atol=1e-10 * np.abs(M).max())


def test_rev_cholesky_kronecker():
    """Section 2: L^(A) (x) L^(B) = RevCholesky(A (x) B)."""
    A, B = _spd(3, 2), _spd(4, 3)
    assert np.allclose(wk.rev_cholesky(np.kron(A, B)),
                       np.kron(wk.rev_cholesky(A), wk.rev_cholesky(B)), atol=1e-12)


def test_waterfilling_worked_example():
    """Figure 1 caption: for L = [[2, 0], [1, 3]] the optimal scales are
    alpha = (3/sqrt(6), 2/sqrt(6)), i.e. Corollary 3.2 with gamma = 1."""
    L = np.array([[2.0, 0.0], [1.0, 3.0]])
    alpha, beta = wk.waterfilling_scales(L, np.array([[1.0]]), 1.0)
    assert np.allclose(alpha, [3 / math.sqrt(6), 2 / math.sqrt(6)], atol=1e-15)
    assert np.allclose(beta, [1.0])
    # the cell is a square of the original volume: alpha_j L_jj equal, product = |L|
    assert np.allclose(alpha * np.diag(L), math.sqrt(6))


def test_normalized_inverse_unit_lower():
    L = wk.rev_cholesky(_spd(12, 4))
    Lt = wk.normalized_inverse(L)
    assert np.allclose(np.diag(Lt), 1.0)
    assert np.allclose(np.triu(Lt, 1), 0.0)
    # columns of L^-1 up to their diagonal scale
    Li = np.linalg.inv(L)
    assert np.allclose(Lt * np.diag(Li)[None, :], Li, atol=1e-12)


def test_two_sided_with_identity_is_gptq():
    """Section 2: with B = I, Algorithm 2 is Algorithm 1."""
    rng = np.random.default_rng(5)
    m, n = 9, 7
    W = rng.standard_normal((m, n))
    A = _spd(n, 6)
    alpha = rng.uniform(0.2, 0.6, n)
    beta = rng.uniform(0.5, 1.5, m)
    Z1 = wk.gptq(W, A, alpha, beta)
    Z2 = wk.gptq2(W, A, np.eye(m), alpha, beta)
    assert np.array_equal(Z1, Z2)


def test_diagonal_geometry_is_plain_rounding():
    """Uncorrelated channels (A, B diagonal): Lt = I, no error feedback, so Z is the
    entrywise rounding of W / (alpha_j beta_i)."""
    rng = np.random.default_rng(7)
    m, n = 8, 6
    W = rng.standard_normal((m, n))
    A = np.diag(rng.uniform(0.5, 2.0, n))
    B = np.diag(rng.uniform(0.5, 2.0, m))
    alpha, beta = rng.uniform(0.1, 0.4, n), rng.uniform(0.5, 1.5, m)
    Z = wk.gptq2(W, A, B, alpha, beta)
    assert np.array_equal(Z, np.rint(W / (beta[:, None] * alpha[None, :])).astype(np.int64))


@pytest.mark.parametrize("seed", [8, 9])
def test_error_in_fundamental_region(seed):
    """Section 2: Algorithm 2 is Babai's nearest plane on the lattice
    (L^A (x) L^B) diag(alpha (x) beta) Z^{mn}, so the transformed error
    E = L^B (V - W) (L^A)^T lies in the box |E_ij| <= alpha_j beta_i L^A_jj L^B_ii / 2."""
    rng = np.random.default_rng(seed)
    m, n = 10, 8
    W = rng.standard_normal((m, n)) * 3.0
    A, B = _spd(n, seed + 10), _spd(m, seed + 20)
    alpha, beta = rng.uniform(0.2, 0.8, n), rng.uniform(0.3, 1.2, m)
    Z = wk.gptq2(W, A, B, alpha, beta)
    V = wk.dequantize(Z, alpha, beta)
    LA, LB = wk.rev_cholesky(A), wk.rev_cholesky(B)
    E = LB @ (V - W) @ LA.T
    box = np.outer(beta * np.diag(LB), alpha * np.diag(LA)) / 2
    assert np.all(np.abs(E) <= box * (1 + 1e-9) + 1e-12)


def test_high_rate_distortion():
    """Corollary 3.2: with the waterfilling scales, D_{A,B} -> gamma^2/12 |A|^(1/n) |B|^(1/m)
    as gamma -> 0 (errors uniform in the cube of side gamma |A|^(1/2n) |B|^(1/2m))."""
    rng = np.random.default_rng(11)
    m, n = 48, 40
    W = rng.standard_normal((m, n))
    A, B = _spd(n, 12, cond=10.0), _spd(m, 13, cond=10.0)
    LA, LB = wk.rev_cholesky(A), wk.rev_cholesky(B)
    gamma = 1e-3
    alpha, beta = wk.waterfilling_scales(LA, LB, gamma)
    Z = wk.gptq2(W, A, B, alpha, beta)
    D = wk.distortion(W, wk.dequantize(Z, alpha, beta), A, B)
    detA = np.exp(np.linalg.slogdet(A)[1] / n)
    detB = np.exp(np.linalg.slogdet(B)[1] / m)
    assert D == pytest.approx(gamma ** 2 / 12 * detA * detB, rel=0.1)


# ---------------------------------------------------------------------------
# planted mistakes in the WaterKron oracle are caught by the pins above
# ---------------------------------------------------------------------------
WK_MUTATIONS = {
    # inverse columns left unnormalised
    "no_normalisation": ("normalized_inverse", lambda L: np.linalg.inv(L)),
    # rows of the inverse normalised instead of columns
    "rows_normalised": ("normalized_inverse",
                        lambda L: (lambda Li: Li / np.diag(Li)[:, None])(
                            np.linalg.inv(L))),
    # ordinary Cholesky (L L^T = M) in place of the reverse one
    "plain_cholesky": ("rev_cholesky", lambda M: np.linalg.cholesky(M)),
}


def _wk_checks():
    return [lambda: test_rev_cholesky_worked_example(),
            lambda: test_rev_cholesky_kronecker(),
            lambda: test_error_in_fundamental_region(8),
            lambda: test_high_rate_distortion()]


@pytest.mark.parametrize("name", sorted(WK_MUTATIONS))
def test_waterkron_mutation_caught(name, monkeypatch):
    attr, fn = WK_MUTATIONS[name]
    monkeypatch.setattr(wk, attr, fn)
    caught = 0
    for check in _wk_checks():
        try:
            check()
        except AssertionError:
            caught += 1
    assert caught > 0, f"mutation {name} not caught by any pin"
