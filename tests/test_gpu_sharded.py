"""Sample-sharded fit through libffh on one GPU: one process holding several shards (the
partial Grams are added on the device; no reduction over processes), compared with the
single-call fit of all samples and with the oracle."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_14706_gb300 as ffh
import synth
from paper_2609_14706_gb300.sharded import fit_sharded

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_14706_gb300 import build
    build.build()


@pytest.mark.parametrize("cuts", [(0, 8192, 16384), (0, 5000, 11111, 16384)])
def test_sharded_fit_matches_single_fit_and_oracle(cuts):
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(N=16384, n=256, m=320, iters=4)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    shards = [(X[a:b], G[a:b]) for a, b in zip(cuts[:-1], cuts[1:])]
    res = fit_sharded(shards, wl.iters)
    with ffh.Handle(dtype="bf16") as h:
        A1, B1 = h.fit(X, G, iters=wl.iters)
    # the same arithmetic up to the order of the fp32 partial sums
    e_self = oracle.kron_rel_err(res.A.cpu(), res.B.cpu(), A1.cpu(), B1.cpu())
    assert e_self < 1e-4, e_self
    ref = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=wl.iters)
    e_ref = oracle.kron_rel_err(res.A.cpu(), res.B.cpu(), ref.A, ref.B)
    assert e_ref <= 2e-3, e_ref
    assert np.trace(oracle.as_f64(res.A)) == pytest.approx(wl.n, rel=1e-4)
    assert res.iters_done == wl.iters and np.isinf(res.deltas[0])


def test_sharded_steps_match_their_definitions():
    """ffh_partial_gram with and without F, accumulation, ffh_update_from_sum with
    damping, ffh_normalize_pair and ffh_relative_change against the oracle."""
    wl = synth.WORKLOADS["tiny_64"].with_(N=3000, n=48, m=40)
    X, G = synth.rank_one_samples(wl, seed=2, device="cuda")
    F = synth.spd_matrix(48, seed=3, cond=100.0, device="cuda")
    Xn, Gn, Fn = oracle.as_f64(X), oracle.as_f64(G), oracle.as_f64(F)
    with ffh.Handle(dtype="f32", damping=0.1) as h:
        P0, ld0 = h.partial_gram(X, G, None)
        P1, ld1 = h.partial_gram(X[:1000], G[:1000], F)
        h.partial_gram(X[1000:], G[1000:], F, P_out=P1, accumulate=True)
        B = h.update_from_sum(P1.clone(), 1.0 / (3000 * 48))
        A = h.update_from_sum(P0[:40, :40].contiguous().clone(), 0.5)[:40, :40].contiguous()
        A2 = A.clone() * 3.0
        s = h.normalize_pair(A2, B)
        dl = h.relative_change(B, P1)
    ref0 = oracle.weighted_gram(Gn, np.einsum("kd,kd->k", Xn, Xn), 1.0)
    w1 = oracle.inv_quad_forms_chol(oracle.cholesky(Fn), Xn)
    ref1 = oracle.weighted_gram(Gn, w1, 1.0)
    # fp32 samples enter the tensor cores as bf16 (both operands): 3 * 2^-9 elementwise
    for got, ref, bound in ((P0, ref0, (np.abs(Gn).T * np.einsum("kd,kd->k", Xn, Xn)) @ np.abs(Gn)),
                            (P1, ref1, (np.abs(Gn).T * w1) @ np.abs(Gn))):
        assert np.all(np.abs(oracle.as_f64(got) - ref) <= 3 * 2.0 ** -9 * bound * 1.05 + 1e-6)
    assert ld0 == 0.0
    assert ld1 == pytest.approx(oracle.logdet_from_cholesky(oracle.cholesky(Fn)), rel=1e-4)
    Bn_ref = oracle.damp(oracle.as_f64(P1) / (3000 * 48), 0.1)
    assert np.allclose(oracle.as_f64(B) / s, Bn_ref, rtol=1e-5, atol=1e-7 * np.abs(Bn_ref).max())
    assert np.trace(oracle.as_f64(A2)) == pytest.approx(40, rel=1e-5)
    assert dl == pytest.approx(oracle.rel_change(oracle.as_f64(B), oracle.as_f64(P1)), rel=1e-4)
