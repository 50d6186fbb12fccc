"""Plant plausible mistakes in the oracle (on the CPU) and check that the pins
catch each one.  This is evidence that the pins constrain every part of the
oracle: a dropped weight, a wrong constant, a wrong inverse, a transposed factor,
swapped roles of x and g, a missing normalisation."""
import numpy as np
import pytest
import scipy.linalg as sla

import oracle
import oracle.flipflop as ff
import test_oracle_pins as pins


def _checks():
    return {
        "factorial": lambda: pins.test_factorial_design_closed_form(),
        "n1": lambda: pins.test_n_equals_one(),
        "m1": lambda: pins.test_m_equals_one(),
        "trace_identity": lambda: pins.test_trace_identity_every_half_step(pins.make_small_fit()),
        "stationary": lambda: pins.test_stationary_equations(pins.make_small_fit()),
        "monotone": lambda: pins.test_loglik_monotone_and_recorded_correctly(pins.make_small_fit()),
        "rademacher": lambda: pins.test_rademacher_identity_input_hessian(),
        "quad_vs_inverse": lambda: pins.test_quad_forms_vs_explicit_inverse(),
        "brute_force": lambda: pins.test_brute_force_minimiser_agrees(),
        "matrix_eq_rank1": lambda: pins.test_matrix_variant_equals_rank_one_variant(),
        "delta_hand": lambda: pins.test_delta_hand_computed_2x2(),
        "delta_invariance": lambda: pins.test_delta_invariant_under_kronecker_rescaling(),
        "delta_iterates": lambda: pins.test_fit_delta_compares_consecutive_iterates(),
        "damped_stationary":
            lambda: pins.test_damped_fixed_point_satisfies_damped_stationary_equations(),
    }


_orig_gram = ff.weighted_gram
_orig_quad = ff.inv_quad_forms_chol
_orig_fit = ff.flipflop_fit
_orig_damp = ff.damp

MUTATIONS = {
    # the weights q_k / r_k are dropped from the Gram
    "dropped_weight": ("weighted_gram", lambda V, w, s: _orig_gram(V, np.ones_like(w), s)),
    # 1/N instead of the MLE constant 1/(N d)
    "wrong_constant": ("weighted_gram", lambda V, w, s: _orig_gram(V, w, 1.0 / V.shape[0])),
    # x^T A x instead of x^T A^-1 x (the Frobenius weights)
    "no_inverse": ("inv_quad_forms_chol", lambda L, V: np.einsum("kd,kd->k", V @ (L @ L.T), V)),
    # forward substitution with L^T read as lower-triangular
    "transposed_factor": ("inv_quad_forms_chol",
                          lambda L, V: (lambda Y: np.einsum("ik,ik->k", Y, Y))(
                              sla.solve_triangular(L.T, V.T, lower=True))),
    # q_k squared (an exponent slip)
    "squared_weight": ("inv_quad_forms_chol", lambda L, V: _orig_quad(L, V) ** 2),
    # delta_t without the trace normalisation of either iterate
    "delta_unnormalised": ("rel_change",
                           lambda F, P: float(np.linalg.norm(F - P) / np.linalg.norm(F))),
    # delta_t relative to the previous iterate instead of the new one
    "delta_old_denominator": ("rel_change", lambda F, P: float(
        np.linalg.norm(F / np.trace(F) - P / np.trace(P)) / np.linalg.norm(P / np.trace(P)))),
    # the damping shift lambda tr(F) instead of lambda mean(diag F)
    "damping_trace_not_mean": ("damp", lambda F, lam: F if lam == 0.0 else
                               F + lam * float(np.trace(F)) * np.eye(F.shape[0])),
}


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, monkeypatch):
    attr, bad = MUTATIONS[name]
    monkeypatch.setattr(ff, attr, bad)
    monkeypatch.setattr(oracle, attr, bad)
    failed = []
    for cname, check in _checks().items():
        try:
            check()
        except (AssertionError, np.linalg.LinAlgError, ValueError, FloatingPointError):
            failed.append(cname)
    assert failed, f"mutation {name} slipped through every pin"


def test_pins_catch_swapped_roles(monkeypatch):
    """x and g exchanged (A fitted from the gradients)."""
    def swapped(X, G, *a, **k):
        r = _orig_fit(G, X, *a, **k)
        r.A, r.B = r.B, r.A
        return r
    monkeypatch.setattr(ff, "flipflop_fit", swapped)
    monkeypatch.setattr(oracle, "flipflop_fit", swapped)
    failed = []
    for cname, check in _checks().items():
        try:
            check()
        except (AssertionError, np.linalg.LinAlgError, ValueError):
            failed.append(cname)
    assert failed


def test_pins_catch_missing_normalisation(monkeypatch):
    """tr(A) = n not enforced (B not carrying the scale)."""
    def unnormalised(X, G, *a, **k):
        r = _orig_fit(X, G, *a, **k)
        r.A = r.A * 3.0
        return r
    monkeypatch.setattr(ff, "flipflop_fit", unnormalised)
    monkeypatch.setattr(oracle, "flipflop_fit", unnormalised)
    failed = []
    for cname, check in _checks().items():
        try:
            check()
        except (AssertionError, np.linalg.LinAlgError, ValueError):
            failed.append(cname)
    assert failed


def _run_checks():
    failed = []
    for cname, check in _checks().items():
        try:
            check()
        except (AssertionError, np.linalg.LinAlgError, ValueError, FloatingPointError):
            failed.append(cname)
    return failed


def test_pins_catch_damping_of_one_factor_only(monkeypatch):
    """Appendix B damps both factors; damping only the B-updates (every other call)."""
    calls = {"n": 0}

    def one_sided(F, lam):
        calls["n"] += 1
        return _orig_damp(F, lam) if calls["n"] % 2 == 1 else F
    monkeypatch.setattr(ff, "damp", one_sided)
    monkeypatch.setattr(oracle, "damp", one_sided)
    assert _run_checks()


def test_pins_catch_damping_only_of_the_returned_pair(monkeypatch):
    """Appendix B damps "including between iterations"; damping only the factors that
    are returned (the iteration itself undamped)."""
    def late(X, G, *a, damping=0.0, **k):
        r = _orig_fit(X, G, *a, **k)
        r.A, r.B = _orig_damp(r.A, damping), _orig_damp(r.B, damping)
        return r
    monkeypatch.setattr(ff, "flipflop_fit", late)
    monkeypatch.setattr(oracle, "flipflop_fit", late)
    assert _run_checks()
