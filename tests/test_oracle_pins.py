"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these re-type the oracle's formulas: each checks the oracle against a
closed form, an invariant, a brute-force evaluation on tiny inputs, or a special
case that reduces to a textbook computation.
"""
import math

import numpy as np
import pytest
import scipy.linalg as sla
import scipy.optimize as so
import torch

import oracle
import synth


def _gauss(N, d, seed, stream=0, scale=1.0):
    return oracle.as_f64(synth.gaussian(N, d, seed=seed, stream=stream, scale=scale))


def _correlated(N, d, seed, stream):
    """Gaussian rows with a seeded non-trivial covariance."""
    S = oracle.as_f64(synth.gaussian(d, d, seed=seed, stream=stream + 50)) / math.sqrt(d)
    S = S + np.eye(d)
    return _gauss(N, d, seed, stream) @ S.T


def _brute_gram(V, w, scale):
    """sum_k w_k v_k v_k^T by explicit outer products."""
    d = V.shape[1]
    C = np.zeros((d, d))
    for k in range(V.shape[0]):
        C += w[k] * np.outer(V[k], V[k])
    return scale * C


def _brute_H(X, G):
    """H = mean_k (x_k (x) g_k)(x_k (x) g_k)^T, formed explicitly (Section 5)."""
    N = X.shape[0]
    H = 0
    for k in range(N):
        v = np.kron(X[k], G[k])
        H = H + np.outer(v, v)
    return H / N


# ---------------------------------------------------------------------------
# single steps
# ---------------------------------------------------------------------------
def test_cholesky_reconstructs_and_logdet():
    A = oracle.as_f64(synth.spd_matrix(9, seed=1, cond=50.0, dtype=torch.float64))
    L = oracle.cholesky(A)
    assert np.allclose(np.triu(L, 1), 0)
    assert np.all(np.diag(L) > 0)
    assert np.allclose(L @ L.T, A, rtol=0, atol=1e-12 * np.abs(A).max())
    # log|A| equals the sum of log-eigenvalues
    assert oracle.logdet_from_cholesky(L) == pytest.approx(
        float(np.sum(np.log(np.linalg.eigvalsh(A)))), rel=1e-12)


def test_tri_inverse_is_inverse():
    A = oracle.as_f64(synth.spd_matrix(11, seed=2, cond=200.0, dtype=torch.float64))
    L = oracle.cholesky(A)
    M = oracle.tri_inverse(L)
    assert np.allclose(np.triu(M, 1), 0)
    assert np.allclose(M @ L, np.eye(11), atol=1e-12)
    assert np.allclose(L @ M, np.eye(11), atol=1e-12)


def test_quad_forms_closed_form_diagonal():
    # A = diag(a): x^T A^-1 x = sum_i x_i^2 / a_i
    a = np.array([0.5, 2.0, 3.0, 7.0, 0.25])
    X = _gauss(13, 5, seed=3)
    q = oracle.inv_quad_forms_chol(np.diag(np.sqrt(a)), X)
    assert np.allclose(q, (X * X / a).sum(1), rtol=1e-13)


def test_quad_forms_vs_explicit_inverse():
    A = oracle.as_f64(synth.spd_matrix(8, seed=4, cond=30.0, dtype=torch.float64))
    X = _gauss(17, 8, seed=4)
    q = oracle.inv_quad_forms_chol(oracle.cholesky(A), X)
    Ainv = np.linalg.inv(A)
    ref = np.array([x @ Ainv @ x for x in X])
    assert np.allclose(q, ref, rtol=1e-11)


def test_weighted_gram_brute_force():
    V = _gauss(23, 6, seed=5)
    w = np.abs(_gauss(23, 1, seed=5, stream=1)[:, 0])
    assert np.allclose(oracle.weighted_gram(V, w, 0.3), _brute_gram(V, w, 0.3), rtol=1e-12)


def test_damp_definition():
    F = np.array([[2.0, 1.0], [1.0, 4.0]])
    D = oracle.damp(F, 0.1)
    assert np.allclose(D, F + 0.3 * np.eye(2))     # 0.1 * mean(2, 4) = 0.3


# ---------------------------------------------------------------------------
# special cases that reduce to textbook results
# ---------------------------------------------------------------------------
def test_rademacher_identity_input_hessian():
    """With B = I and g_k in {+-1}^m, one A-update is X^T X / N (the input-only GPTQ
    Hessian, Table 1 'Input')."""
    N, n, m = 300, 7, 5
    X = _correlated(N, n, seed=6, stream=0)
    G = oracle.as_f64(synth.rademacher(N, m, seed=6))
    r = oracle.inv_quad_forms_chol(np.eye(m), G)             # g^T I^-1 g = m
    A = oracle.weighted_gram(X, r, 1.0 / (N * m))
    ref = np.zeros((n, n))
    for k in range(N):
        ref += np.outer(X[k], X[k])
    assert np.allclose(A, ref / N, rtol=1e-12)
    A_in, B_in = oracle.input_hessian(X, m)
    assert np.allclose(A_in, ref / N, rtol=1e-12) and np.allclose(B_in, np.eye(m))


def test_factorial_design_closed_form():
    """All P*R pairs of P inputs and R gradients: H = Sigma_x (x) Sigma_g exactly, and
    the fit reaches A = n Sigma_x / tr Sigma_x, B = (tr Sigma_x / n) Sigma_g after one
    iteration (mean_p x_p^T Sigma_x^-1 x_p = n), then stays there."""
    P, R, n, m = 12, 9, 5, 4
    X, G, Xp, Gr = synth.factorial_design(P, R, n, m, seed=7, dtype=torch.float64)
    Xp, Gr = oracle.as_f64(Xp), oracle.as_f64(Gr)
    Sx = sum(np.outer(x, x) for x in Xp) / P
    Sg = sum(np.outer(g, g) for g in Gr) / R
    fit = oracle.flipflop_fit(X, G, iters=1)
    assert np.allclose(fit.A, n * Sx / np.trace(Sx), rtol=1e-11)
    assert np.allclose(fit.B, np.trace(Sx) / n * Sg, rtol=1e-11)
    fit3 = oracle.flipflop_fit(X, G, iters=3)
    assert np.allclose(np.kron(fit3.A, fit3.B), np.kron(Sx, Sg), rtol=1e-10)
    assert fit3.deltas[1] < 1e-12 and fit3.deltas[2] < 1e-12


def test_n_equals_one():
    """n = 1: A is a scalar, A = 1 after normalisation and B = E[x^2 g g^T] exactly
    after one iteration."""
    N, m = 200, 6
    x = _gauss(N, 1, seed=8)
    G = _correlated(N, m, seed=8, stream=1)
    fit = oracle.flipflop_fit(x, G, iters=2)
    ref = sum(x[k, 0] ** 2 * np.outer(G[k], G[k]) for k in range(N)) / N
    assert fit.A.shape == (1, 1) and fit.A[0, 0] == pytest.approx(1.0, rel=1e-13)
    assert np.allclose(fit.B, ref, rtol=1e-11)


def test_m_equals_one():
    """m = 1: the fixed point is A (x) B = E[g^2 x x^T] (reached after two
    iterations from A_0 = I)."""
    N, n = 200, 6
    X = _correlated(N, n, seed=9, stream=0)
    g = _gauss(N, 1, seed=9, stream=1)
    fit = oracle.flipflop_fit(X, g, iters=3)
    ref = sum(g[k, 0] ** 2 * np.outer(X[k], X[k]) for k in range(N)) / N
    assert np.allclose(fit.A * fit.B[0, 0], ref, rtol=1e-11)
    assert np.trace(fit.A) == pytest.approx(n, rel=1e-13)


# ---------------------------------------------------------------------------
# invariants
# ---------------------------------------------------------------------------
def make_small_fit():
    N, n, m = 400, 6, 5
    X = _correlated(N, n, seed=10, stream=0)
    G = _correlated(N, m, seed=10, stream=1)
    # make x and g dependent, so H is not a Kronecker product
    G = G * (1.0 + 0.5 * np.abs(X[:, :1]))
    return X, G, oracle.flipflop_fit(X, G, iters=40)


@pytest.fixture(scope="module")
def small_fit():
    return make_small_fit()


def test_trace_identity_every_half_step(small_fit):
    """mean_k q_k r_k = m n after every undamped half-step (trace of the update)."""
    X, G, fit = small_fit
    n, m = X.shape[1], G.shape[1]
    assert np.allclose(fit.mean_qr, m * n, rtol=1e-10)


def test_loglik_monotone_and_recorded_correctly(small_fit):
    """Each half-step is an exact block minimiser (Section 5), so the Gaussian
    log-likelihood never decreases (Section 4 KL relation)."""
    X, G, fit = small_fit
    ll = np.array(fit.loglik)
    assert np.all(np.diff(ll) >= -1e-9 * np.abs(ll[:-1]))
    assert ll[-1] > ll[0]
    # the recorded final value equals a from-scratch evaluation at (A, B)
    assert oracle.loglik(X, G, fit.A, fit.B) == pytest.approx(ll[-1], rel=1e-10)


def test_phi_tilde_monotone():
    N, n, m = 300, 5, 4
    X = _correlated(N, n, seed=11, stream=0)
    G = _correlated(N, m, seed=11, stream=1) * (1 + np.abs(X[:, 1:2]))
    phis = [oracle.phi_tilde(X, G, *oracle.marginal_hessian(X, G))]
    for it in range(1, 8):
        f = oracle.flipflop_fit(X, G, iters=it)
        phis.append(oracle.phi_tilde(X, G, f.A, f.B))
    assert np.all(np.diff(phis[1:]) <= 1e-12)
    # FlipFlop beats the Marginal Hessian on its own objective
    assert phis[-1] <= phis[0] + 1e-12


def test_stationary_equations(small_fit):
    """At convergence A propto E[(g^T B^-1 g) x x^T] and B propto E[(x^T A^-1 x) g g^T]
    with the MLE constants (Section 5 fixed-point equations)."""
    X, G, fit = small_fit
    N, n = X.shape
    m = G.shape[1]
    Ai, Bi = np.linalg.inv(fit.A), np.linalg.inv(fit.B)
    q = np.array([x @ Ai @ x for x in X])
    r = np.array([g @ Bi @ g for g in G])
    A_rhs = _brute_gram(X, r, 1.0 / (N * m))
    B_rhs = _brute_gram(G, q, 1.0 / (N * n))
    assert np.linalg.norm(fit.A - A_rhs) / np.linalg.norm(fit.A) < 1e-9
    assert np.linalg.norm(fit.B - B_rhs) / np.linalg.norm(fit.B) < 1e-9


def test_damping_breaks_trace_identity_as_expected():
    N, n, m = 200, 4, 3
    X = _correlated(N, n, seed=12, stream=0)
    G = _correlated(N, m, seed=12, stream=1)
    f = oracle.flipflop_fit(X, G, iters=3, damping=0.1)
    assert not np.allclose(f.mean_qr, m * n, rtol=1e-6)
    # damped factors are what the next step inverts: B's diagonal got the shift
    f1 = oracle.flipflop_fit(X, G, iters=1, damping=0.0)
    assert np.trace(f.B) != pytest.approx(np.trace(f1.B), rel=1e-6)


def test_delta_hand_computed_2x2():
    """delta_t's definition worked by hand: A_t = diag(2, 1), A_{t-1} = I_2 give
    A^_t = diag(2/3, 1/3), A^_{t-1} = diag(1/2, 1/2), difference diag(1/6, -1/6) with
    norm sqrt(2)/6, ||A^_t|| = sqrt(5)/3, so delta = 1/sqrt(10).  A missing trace
    normalisation gives 1/sqrt(5), the norm of A^_{t-1} in the denominator 1/3."""
    At = np.diag([2.0, 1.0])
    Ap = np.eye(2)
    assert oracle.rel_change(At, Ap) == pytest.approx(1.0 / math.sqrt(10.0), rel=1e-15)
    # an off-diagonal pair: A_t = [[3, 1], [1, 1]] (tr 4), A_{t-1} = [[1, 0], [0, 3]]
    # (tr 4): difference [[2, 1], [1, -2]] / 4, norm sqrt(10)/4; ||A^_t|| = sqrt(12)/4
    At = np.array([[3.0, 1.0], [1.0, 1.0]])
    Ap = np.array([[1.0, 0.0], [0.0, 3.0]])
    assert oracle.rel_change(At, Ap) == pytest.approx(math.sqrt(10.0 / 12.0), rel=1e-15)


def test_delta_invariant_under_kronecker_rescaling():
    """The fixed point is defined only up to (c A, B / c) (Section 5), so delta must not
    change when either iterate of either factor is rescaled."""
    rng = np.random.default_rng(21)
    for _ in range(5):
        a = rng.standard_normal((4, 4))
        b = rng.standard_normal((4, 4))
        F, P = a @ a.T + np.eye(4), b @ b.T + np.eye(4)
        ref = oracle.rel_change(F, P)
        for c1, c2 in ((3.0, 1.0), (1.0, 0.2), (7.5, 1e-3)):
            assert oracle.rel_change(c1 * F, c2 * P) == pytest.approx(ref, rel=1e-13)


def test_fit_delta_compares_consecutive_iterates():
    """The fit's recorded delta_t is the larger of the two factors' changes between the
    iterates it returned after t-1 and t iterations (the first is +inf), and it goes
    to zero at a fixed point: the factorial design reaches its closed form in one
    iteration (see test_factorial_design_closed_form), so delta_2 = delta_3 = 0."""
    X, G, _ = make_small_fit()
    f = oracle.flipflop_fit(X, G, iters=6, keep_iterates=True)
    assert math.isinf(f.deltas[0])
    for t in range(1, 6):
        (A1, B1), (A0, B0) = f.iterates[t], f.iterates[t - 1]
        want = max(oracle.rel_change(A1, A0), oracle.rel_change(B1, B0))
        assert f.deltas[t] == pytest.approx(want, rel=1e-12)
    # the same iterates come back from fits of fewer iterations
    f3 = oracle.flipflop_fit(X, G, iters=3)
    assert np.allclose(f3.A, f.iterates[2][0], rtol=1e-12)
    assert np.allclose(f3.B, f.iterates[2][1], rtol=1e-12)
    Xf, Gf, _, _ = synth.factorial_design(8, 7, 4, 3, seed=22, dtype=torch.float64)
    ff3 = oracle.flipflop_fit(Xf, Gf, iters=3)
    assert max(ff3.deltas[1:]) < 1e-13


def test_damped_fixed_point_satisfies_damped_stationary_equations():
    """With damping lambda > 0 (Appendix B: each factor is damped when it is computed,
    including between iterations) the iteration converges to a pair with
        A propto damp(E[(g^T B^-1 g) x x^T], lambda),  B propto damp(E[(x^T A^-1 x) g g^T], lambda),
    damp(F) = F + lambda mean(diag F) I, checked by brute force (explicit inverses and
    outer products) at the returned pair, each equation up to a positive scale."""
    N, n, m = 300, 5, 4
    X = _correlated(N, n, seed=23, stream=0)
    G = _correlated(N, m, seed=23, stream=1) * (1.0 + 0.7 * np.abs(X[:, 2:3]))
    lam = 0.1
    fit = oracle.flipflop_fit(X, G, iters=400, damping=lam)
    assert fit.deltas[-1] < 1e-13
    Ai, Bi = np.linalg.inv(fit.A), np.linalg.inv(fit.B)
    q = np.array([x @ Ai @ x for x in X])
    r = np.array([g @ Bi @ g for g in G])

    def damped(F):
        return F + lam * np.trace(F) / F.shape[0] * np.eye(F.shape[0])

    A_rhs = damped(_brute_gram(X, r, 1.0))
    B_rhs = damped(_brute_gram(G, q, 1.0))
    for F, R in ((fit.A, A_rhs), (fit.B, B_rhs)):
        Fh, Rh = F / np.trace(F), R / np.trace(R)
        assert np.linalg.norm(Fh - Rh) / np.linalg.norm(Rh) < 1e-10
    # the undamped stationary equations do not hold there
    Ah = _brute_gram(X, r, 1.0)
    assert np.linalg.norm(fit.A / np.trace(fit.A) - Ah / np.trace(Ah)) > 1e-4
    # and the damped fixed point differs from the undamped one
    f0 = oracle.flipflop_fit(X, G, iters=400)
    assert oracle.kron_rel_err(fit.A, fit.B, f0.A, f0.B) > 1e-3


def test_damping_is_homogeneous_so_it_commutes_with_the_rescale():
    """damp(c F) = c damp(F) for c > 0: damping before or after the tr(A) = n rescale
    gives the same pair, so the order of those two steps is not a reading that
    matters; the one that does (damping inside the iteration, before the next
    inversion) is pinned by the damped stationary equations above."""
    F = np.array([[2.0, 0.5, 0.1], [0.5, 3.0, 0.2], [0.1, 0.2, 1.0]])
    for c in (0.3, 2.0, 17.0):
        assert np.allclose(oracle.damp(c * F, 0.1), c * oracle.damp(F, 0.1), rtol=1e-15)


def test_row_blocks_do_not_change_the_fit():
    """The expectations are accumulated over blocks of rows; any block size gives the
    same fit (up to the order of the additions), including a ragged last block."""
    X, G, _ = make_small_fit()
    f_all = oracle.flipflop_fit(X, G, iters=5)
    f_7 = oracle.flipflop_fit(X, G, iters=5, rows=7)
    f_64 = oracle.flipflop_fit(X, G, iters=5, rows=64)
    def rel(P, Q):
        return np.linalg.norm(P - Q) / np.linalg.norm(Q)

    for f in (f_7, f_64):
        assert rel(f.A, f_all.A) < 1e-12 and rel(f.B, f_all.B) < 1e-12
        assert np.allclose(f.loglik, f_all.loglik, rtol=1e-12)
    # bf16 samples held as torch tensors are widened block by block
    Xb = torch.from_numpy(X).to(torch.bfloat16)
    Gb = torch.from_numpy(G).to(torch.bfloat16)
    fb = oracle.flipflop_fit(Xb, Gb, iters=3, rows=33)
    fr = oracle.flipflop_fit(oracle.as_f64(Xb), oracle.as_f64(Gb), iters=3)
    assert rel(fb.A, fr.A) < 1e-12 and rel(fb.B, fr.B) < 1e-12


def test_matrix_fit_over_sample_blocks_equals_matrix_fit():
    """The block-accumulated matrix fit (samples drawn block by block) is the same fit:
    sums over samples grouped differently, including a ragged last block."""
    N, m, n = 37, 5, 4
    rng = np.random.default_rng(31)
    Gk = rng.standard_normal((N, m, n)) * (1.0 + np.abs(rng.standard_normal((N, 1, 1))))
    ref = oracle.flipflop_fit_matrix(Gk, iters=6, damping=0.05)

    def blocks():
        for k0 in range(0, N, 10):
            yield Gk[k0:k0 + 10]

    A, B, t, deltas = oracle.flipflop_fit_matrix_blocks(blocks, N, m, n, iters=6, damping=0.05)
    assert t == 6
    assert np.linalg.norm(A - ref.A) / np.linalg.norm(ref.A) < 1e-12
    assert np.linalg.norm(B - ref.B) / np.linalg.norm(ref.B) < 1e-12
    assert np.allclose(deltas[1:], ref.deltas[1:], rtol=1e-8)


def test_tol_stops_early():
    N, n, m = 300, 4, 3
    X = _correlated(N, n, seed=13, stream=0)
    G = _correlated(N, m, seed=13, stream=1)
    f = oracle.flipflop_fit(X, G, iters=200, tol=1e-6)
    assert f.iters_done < 200 and f.deltas[-1] < 1e-6
    assert all(d >= 1e-6 for d in f.deltas[:-1])
    assert math.isinf(f.deltas[0])


# ---------------------------------------------------------------------------
# brute force on tiny inputs
# ---------------------------------------------------------------------------
def _phi_full(H, A, B):
    """Phi(H, A (x) B) from its definition (Section 4), with |H| included."""
    n, m = A.shape[0], B.shape[0]
    K = np.kron(A, B)
    tr = np.trace(H @ np.linalg.inv(K)) / (m * n)
    ldH = np.linalg.slogdet(H)[1]
    return tr / math.exp(ldH / (m * n) - np.linalg.slogdet(A)[1] / n - np.linalg.slogdet(B)[1] / m)


def test_phi_is_am_over_gm_of_generalized_eigenvalues():
    N, n, m = 60, 3, 2
    X = _correlated(N, n, seed=14, stream=0)
    G = _correlated(N, m, seed=14, stream=1) * (1 + np.abs(X[:, :1]))
    H = _brute_H(X, G)
    A, B = oracle.marginal_hessian(X, G)
    lam = sla.eigh(H, np.kron(A, B), eigvals_only=True)
    am, gm = lam.mean(), math.exp(np.mean(np.log(lam)))
    assert _phi_full(H, A, B) == pytest.approx(am / gm, rel=1e-10)
    # the sample form |A|^{1/n}|B|^{1/m} mean(q r)/(mn) is Phi * |H|^{1/mn}
    phi_t = oracle.phi_tilde(X, G, A, B)
    assert phi_t == pytest.approx(am / gm * math.exp(np.linalg.slogdet(H)[1] / (m * n)), rel=1e-9)


def test_brute_force_minimiser_agrees():
    """Minimise log Phi over A, B (Cholesky parameters) with a generic optimiser on
    an explicitly formed H; the flip-flop fixed point must attain the minimum."""
    N, n, m = 80, 3, 2
    X = _correlated(N, n, seed=15, stream=0)
    G = _correlated(N, m, seed=15, stream=1) * (1 + 0.7 * np.abs(X[:, :1]))
    H = _brute_H(X, G)
    il_a, il_b = np.tril_indices(n), np.tril_indices(m)

    def unpack(p):
        La = np.zeros((n, n))
        La[il_a] = p[: len(il_a[0])]
        Lb = np.zeros((m, m))
        Lb[il_b] = p[len(il_a[0]):]
        La[np.diag_indices(n)] = np.exp(np.diag(La))
        Lb[np.diag_indices(m)] = np.exp(np.diag(Lb))
        return La @ La.T, Lb @ Lb.T

    def objective(p):
        A, B = unpack(p)
        K = np.kron(A, B)
        return (math.log(np.trace(np.linalg.solve(K, H)) / (m * n))
                + np.linalg.slogdet(A)[1] / n + np.linalg.slogdet(B)[1] / m)

    p0 = np.zeros(len(il_a[0]) + len(il_b[0]))
    res = so.minimize(objective, p0, method="BFGS", options={"gtol": 1e-11, "maxiter": 10000})
    A_bf, B_bf = unpack(res.x)
    fit = oracle.flipflop_fit(X, G, iters=300, tol=1e-14)
    p_ff = math.log(_phi_full(H, fit.A, fit.B))
    p_bf = math.log(_phi_full(H, A_bf, B_bf))
    assert p_ff <= p_bf + 1e-10
    assert abs(p_ff - p_bf) < 1e-7
    assert oracle.kron_rel_err(fit.A, fit.B, A_bf, B_bf) < 1e-4
    assert _phi_full(H, fit.A, fit.B) >= 1.0


def test_phi_equals_one_iff_kronecker():
    """Phi = 1 exactly when H = A (x) B (factorial design makes H Kronecker)."""
    P, R, n, m = 7, 6, 3, 2
    X, G, _, _ = synth.factorial_design(P, R, n, m, seed=16, dtype=torch.float64)
    X, G = oracle.as_f64(X), oracle.as_f64(G)
    H = _brute_H(X, G)
    fit = oracle.flipflop_fit(X, G, iters=2)
    assert _phi_full(H, fit.A, fit.B) == pytest.approx(1.0, abs=1e-10)
    assert _phi_full(H, np.eye(n), np.eye(m)) > 1.0 + 1e-3


def test_matrix_variant_equals_rank_one_variant():
    """G_k = g_k x_k^T turns the matrix-sample updates into the rank-one updates."""
    N, n, m = 150, 5, 4
    X = _correlated(N, n, seed=17, stream=0)
    G = _correlated(N, m, seed=17, stream=1) * (1 + np.abs(X[:, :1]))
    Gk = np.einsum("ki,kj->kij", G, X)
    f1 = oracle.flipflop_fit(X, G, iters=5)
    f2 = oracle.flipflop_fit_matrix(Gk, iters=5)
    assert np.allclose(f1.A, f2.A, rtol=1e-10) and np.allclose(f1.B, f2.B, rtol=1e-10)
    assert np.allclose(f1.loglik, f2.loglik, rtol=1e-10)


# ---------------------------------------------------------------------------
# population recovery
# ---------------------------------------------------------------------------
def test_recovery_rank_one_rate():
    """x independent of g: H -> Sigma_x (x) Sigma_g, so the fit approaches the
    population product at rate N^-1/2."""
    n, m = 8, 6
    Sx = oracle.as_f64(synth.spd_matrix(n, seed=18, cond=20.0, dtype=torch.float64))
    Sg = oracle.as_f64(synth.spd_matrix(m, seed=19, cond=10.0, dtype=torch.float64))
    Lx, Lg = np.linalg.cholesky(Sx), np.linalg.cholesky(Sg)
    errs = []
    for N in (1000, 100000):
        X = _gauss(N, n, seed=20, stream=0) @ Lx.T
        G = _gauss(N, m, seed=20, stream=1) @ Lg.T
        f = oracle.flipflop_fit(X, G, iters=30, tol=1e-12)
        errs.append(oracle.kron_rel_err(f.A, f.B, Sx, Sg))
    assert errs[1] < errs[0] / 4.0     # sqrt(100) = 10 expected
    assert errs[1] < 0.02


def test_recovery_matrix_normal():
    wl = synth.WORKLOADS["kron_recovery_512x768"].with_(n=6, m=5)
    _, _, A0, B0 = synth.matrix_normal_factors(wl, seed=0)
    errs = []
    for N in (200, 20000):
        Gk = synth.matrix_samples(wl, seed=0, N=N)
        f = oracle.flipflop_fit_matrix(Gk, iters=30, tol=1e-12)
        errs.append(oracle.kron_rel_err(f.A, f.B, A0, B0))
    assert errs[1] < errs[0] / 4.0
    assert errs[1] < 0.02


# ---------------------------------------------------------------------------
# comparison variants and the parity metric
# ---------------------------------------------------------------------------
def test_frobenius_variant_reaches_van_loan_pitsianis_optimum():
    """The Frobenius Hessian iteration converges to the best Kronecker approximation
    in Frobenius norm: the top singular pair of the rearranged H."""
    N, n, m = 120, 3, 2
    X = _correlated(N, n, seed=21, stream=0)
    G = _correlated(N, m, seed=21, stream=1) * (1 + np.abs(X[:, :1]))
    # rearrangement R(H) = mean_k vec(x x^T) vec(g g^T)^T  (n^2 x m^2)
    R = sum(np.outer(np.outer(x, x).ravel(), np.outer(g, g).ravel()) for x, g in zip(X, G)) / N
    U, s, Vt = np.linalg.svd(R)
    A_opt = (s[0] * U[:, 0]).reshape(n, n)
    B_opt = Vt[0].reshape(m, m)
    f = oracle.frobenius_fit(X, G, iters=200)
    assert np.allclose(np.kron(f.A, f.B), np.kron(A_opt, B_opt), rtol=1e-8, atol=1e-10)


def test_kron_metric_closed_form_matches_explicit():
    rng = np.random.default_rng(0)
    A, A2 = (oracle.as_f64(synth.spd_matrix(4, seed=s, dtype=torch.float64)) for s in (30, 31))
    B, B2 = (oracle.as_f64(synth.spd_matrix(3, seed=s, dtype=torch.float64)) for s in (32, 33))
    a, b, a2, b2 = (F / np.trace(F) for F in (A, B, A2, B2))
    ref = np.linalg.norm(np.kron(a, b) - np.kron(a2, b2)) / np.linalg.norm(np.kron(a2, b2))
    assert oracle.kron_rel_err(A, B, A2, B2) == pytest.approx(ref, rel=1e-10)
    c = float(rng.uniform(0.1, 10))
    assert oracle.kron_rel_err(c * A, B / c, A, B) < 1e-7
