"""Parity at the full workload sizes, in the configuration bench.py times.

The oracle cannot run whole fits at these sizes in a test, so it checks outputs it can
compute one by one (sampled entries of the first B-update and of weighted Grams,
sampled quadratic forms, sampled columns of Cholesky residuals), and the fits are
checked through properties that hold at any size (trace identity, monotone
log-likelihood, tr A = n, symmetry, positive definiteness).
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2609_14706_gb300 as ffh
import synth

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

RANK_ONE = ["llama7b_attn_4096", "llama7b_mlp_up_4096x11008", "llama3_8b_down_14336x4096"]


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_14706_gb300 import build
    build.build()


def _free_gb():
    free, _ = torch.cuda.mem_get_info()
    return free / 1e9


def _is_spd(F):
    """Positive definiteness by an independent fp64 Cholesky (torch)."""
    _, info = torch.linalg.cholesky_ex(F.double().cpu())
    return int(info) == 0


def _row_norms_f64(V, chunk=4096):
    """||v_k||^2 in fp64 on the host, chunk by chunk."""
    out = np.empty(V.shape[0])
    for r0 in range(0, V.shape[0], chunk):
        v = oracle.as_f64(V[r0:r0 + chunk])
        out[r0:r0 + chunk] = np.einsum("kd,kd->k", v, v)
    return out


@pytest.mark.parametrize("name", RANK_ONE)
def test_first_b_update_sampled_entries(name):
    """One iteration from A_0 = I: B_1 = 1/(N n) sum_k ||x_k||^2 g_k g_k^T (Section 5 with
    A = I).  The returned B is B_1 times the normalisation factor, so ratios of sampled
    entries to a sampled diagonal entry are compared (scale-free)."""
    wl = synth.WORKLOADS[name]
    if _free_gb() < 3 * wl.sample_bytes() / 1e9 + 8:
        pytest.skip("not enough free device memory")
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16") as h:
        A, B = h.fit(X, G, iters=1)
    torch.cuda.synchronize()
    q = _row_norms_f64(X)
    rng = np.random.default_rng(1)
    idx = np.unique(rng.integers(0, wl.m, 24))
    Gs = oracle.as_f64(G[:, torch.as_tensor(idx, device="cuda")])
    Bs = oracle.as_f64(B[torch.as_tensor(idx, device="cuda")][:, torch.as_tensor(idx, device="cuda")])
    ref = (Gs.T * q) @ Gs / (wl.N * wl.n)
    # entries relative to the first sampled diagonal entry
    got, want = Bs / Bs[0, 0], ref / ref[0, 0]
    scale = np.sqrt(np.outer(np.diag(want), np.diag(want)))
    assert np.max(np.abs(got - want) / scale) <= 4e-3
    # A_1 itself: tr A = n, symmetric
    An = oracle.as_f64(A)
    assert np.trace(An) == pytest.approx(wl.n, rel=1e-4)
    assert np.array_equal(An, An.T)


@pytest.mark.parametrize("name", RANK_ONE)
def test_full_fit_properties(name):
    """Full fit (all iterations): trace identity mean_k q_k r_k = m n after every
    half-step, non-decreasing log-likelihood, tr A = n, symmetric positive definite."""
    wl = synth.WORKLOADS[name]
    if _free_gb() < 3 * wl.sample_bytes() / 1e9 + 8:
        pytest.skip("not enough free device memory")
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16", final_loglik=True) as h:
        A, B = h.fit(X, G, iters=wl.iters)
        st = h.stats()
    assert st["iters_done"] == wl.iters
    assert np.allclose(st["mean_qr"], wl.m * wl.n, rtol=2e-2)
    ll = np.array(st["loglik"])
    assert np.all(np.isfinite(ll))
    # monotone up to the rounding of the bf16 passes (relative 1e-5 of |l|)
    assert np.all(np.diff(ll) >= -1e-5 * np.abs(ll[:-1]))
    An, Bn = oracle.as_f64(A), oracle.as_f64(B)
    assert np.trace(An) == pytest.approx(wl.n, rel=1e-4)
    assert np.array_equal(An, An.T) and np.array_equal(Bn, Bn.T)
    assert np.all(np.isfinite(An)) and np.all(np.isfinite(Bn))
    assert _is_spd(A) and _is_spd(B)


@pytest.mark.parametrize("d", [4096, 11008, 14336])
def test_weighted_gram_sampled_entries_full_size(d):
    """Sampled entries of scale * V^T diag(w) V at N = 262144 (the headline length),
    each computed by the oracle as one fp64 dot product over the samples."""
    N = 262144
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(n=d, m=8)
    X, _ = synth.rank_one_samples(wl, seed=2, device="cuda", N=N)
    w = torch.rand(N, device="cuda", generator=torch.Generator("cuda").manual_seed(3)) + 0.25
    scale = 1.0 / (N * 7)
    with ffh.Handle(dtype="bf16") as h:
        C = h.weighted_gram(X, w, scale)
    torch.cuda.synchronize()
    rng = np.random.default_rng(4)
    pairs = np.stack([rng.integers(0, d, 48), rng.integers(0, d, 48)], 1)
    cols = np.unique(pairs)
    Vc = oracle.as_f64(X[:, torch.as_tensor(cols, device="cuda")])
    wn = oracle.as_f64(w)
    pos = {c: i for i, c in enumerate(cols)}
    Cn = C.cpu()
    for i, j in pairs:
        a, b = Vc[:, pos[i]], Vc[:, pos[j]]
        ref = scale * np.dot(wn * a, b)
        bound = 2.0 ** -8 * scale * np.dot(wn * np.abs(a), np.abs(b))
        assert abs(float(Cn[i, j]) - ref) <= bound + 1e-7 * abs(ref)
        assert float(Cn[i, j]) == float(Cn[j, i])


def test_quad_form_sampled_rows_full_size():
    """Sampled q_k = x_k^T A^-1 x_k at n = 4096, N = 262144 (oracle: forward
    substitution with its own fp64 Cholesky factor)."""
    wl = synth.WORKLOADS["llama7b_attn_4096"]
    X, _ = synth.rank_one_samples(wl.with_(m=8), seed=5, device="cuda")
    A = oracle.as_f64(synth.spd_matrix(wl.n, seed=6, cond=1e3, dtype=torch.float64))
    Lr = oracle.cholesky(A)
    Mr = oracle.tri_inverse(Lr)
    with ffh.Handle(dtype="bf16") as h:
        q = h.quad_form(X, torch.tensor(Mr, dtype=torch.float32, device="cuda"))
    rows = np.random.default_rng(7).integers(0, wl.N, 64)
    Xs = oracle.as_f64(X[torch.as_tensor(rows, device="cuda")])
    ref = oracle.inv_quad_forms_chol(Lr, Xs)
    Mf = Mr.astype(np.float32).astype(np.float64)
    y, z = Xs @ Mf.T, np.abs(Xs) @ np.abs(Mf).T
    bound = (2.0 ** -8 * np.sum(np.abs(y) * z, 1) + 2.0 ** -18 * np.sum(z * z, 1) + 1e-5 * ref
             + np.abs(np.sum(y * y, 1) - ref))
    assert np.all(np.abs(oracle.as_f64(q)[rows] - ref) <= bound)


@pytest.mark.parametrize("d", [11008, 14336])
def test_cholesky_sampled_columns_full_size(d):
    """Backward error and inverse residual on sampled columns at the largest factor
    sizes: ||(L L^T - F) e_j|| and ||(M L - I) e_j|| for 16 columns j."""
    F = synth.spd_matrix(d, seed=8, cond=1e3, dtype=torch.float32, device="cuda")
    with ffh.Handle() as h:
        L, M, logdet = h.cholesky(F)
    cols = np.random.default_rng(9).integers(0, d, 16)
    Lh = oracle.as_f64(L)
    Mh = oracle.as_f64(M)
    Fh = oracle.as_f64(F)
    u_eff = 2.0 ** -16
    for j in cols:
        back = np.linalg.norm(Lh @ Lh[j] - Fh[:, j]) / np.linalg.norm(Fh[:, j])
        e = np.zeros(d)
        e[j] = 1.0
        inv = np.linalg.norm(Mh @ Lh[:, j] - e)
        assert back <= 64 * u_eff, (j, back)
        assert inv <= 8 * u_eff * math.sqrt(1e3) * math.sqrt(d), (j, inv)
    assert np.isfinite(logdet)


def test_matrix_fit_full_size():
    """The Kronecker ground-truth recovery workload at full size (N = 65536 matrix samples,
    n = 512, m = 768, 20 iterations): tr A = n, SPD, non-decreasing log-likelihood, and
    the fit recovers the population A0 (x) B0 (the MLE error at this N is small)."""
    wl = synth.WORKLOADS["kron_recovery_512x768"]
    need = wl.sample_bytes() * 1.6 / 1e9 + 8
    if _free_gb() < need:
        pytest.skip(f"needs about {need:.0f} GB of free device memory")
    Gk = synth.matrix_samples(wl, seed=0, device="cuda")
    _, _, A0, B0 = synth.matrix_normal_factors(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="f32", final_loglik=True) as h:
        A, B = h.fit_matrix(Gk, iters=wl.iters)
        st = h.stats()
    del Gk
    torch.cuda.empty_cache()
    ll = np.array(st["loglik"])
    assert np.all(np.diff(ll) >= -1e-5 * np.abs(ll[:-1]))
    assert np.trace(oracle.as_f64(A)) == pytest.approx(wl.n, rel=1e-4)
    assert _is_spd(A) and _is_spd(B)
    err = oracle.kron_rel_err(A.cpu(), B.cpu(), A0.cpu(), B0.cpu())
    assert err < 0.05, err
