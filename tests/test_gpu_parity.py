"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

Tolerances are derived from the arithmetic of each step:
  * weighted Gram: the weighted operand is rounded to bf16 once (relative error
    <= 2^-9 per term) and accumulated in fp32, so elementwise
    |C - C_ref| <= 2^-8 * (|V|^T diag(|w|) |V|) * scale   (2^-8 leaves room for the
    fp32 accumulation, whose error is orders of magnitude smaller for N <= 2^19);
  * quadratic form: L^-1 is rounded to bf16 (2^-9 per entry), inputs are exact,
    so with y = L^-1 v, z = |L^-1| |v|:  |q - q_ref| <= 2^-8 sum_i |y_i| z_i
    + 2^-18 sum_i z_i^2 (plus fp32 accumulation);
  * the fit: relative Frobenius error of the trace-normalised A (x) B <= 2e-3.
"""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2609_14706_gb300 as ffh
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_14706_gb300 import build
    build.build()


def _bf16_gram_bound(V, w, scale):
    Va = np.abs(V)
    wa = np.ones(V.shape[0]) if w is None else np.abs(w)
    return 2.0 ** -8 * scale * ((Va.T * wa) @ Va)


# ---------------------------------------------------------------------------
# weighted Gram
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N,d,weighted", [(1000, 64, True), (5000, 320, True), (4097, 136, False),
                                          (3000, 512, True), (700, 8, True)])
def test_weighted_gram_matches_oracle(N, d, weighted):
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(n=d, m=8)
    X, _ = synth.rank_one_samples(wl, seed=1, device="cuda", N=N)
    w = (torch.rand(N, device="cuda", generator=torch.Generator("cuda").manual_seed(2)) * 3
         if weighted else None)
    scale = 1.0 / (N * 7)
    with ffh.Handle(dtype="bf16") as h:
        C = h.weighted_gram(X, w, scale)
    torch.cuda.synchronize()
    Vn = oracle.as_f64(X)
    wn = None if w is None else oracle.as_f64(w)
    ref = oracle.weighted_gram(Vn, np.ones(N) if wn is None else wn, scale)
    Cn = oracle.as_f64(C)
    assert np.array_equal(Cn, Cn.T), "output must be exactly symmetric"
    bound = _bf16_gram_bound(Vn, wn, scale) + 1e-7 * np.abs(ref).max()
    assert np.all(np.abs(Cn - ref) <= bound), np.max(np.abs(Cn - ref) / bound)


@pytest.mark.parametrize("N,d", [(2048, 4096), (4097, 4096), (9000, 4096), (5000, 4000)])
def test_weighted_gram_headline_width_matches_oracle(N, d):
    """The headline width (d = 4096, and a partial last tile at 4000) with several sample
    blocks and a ragged N: elementwise bound, determinism, exact symmetry, and the relative
    Frobenius error, which is what the fit's accuracy depends on (a single fp32 TMEM
    accumulator over very many samples stays inside the elementwise bound while losing an
    order of magnitude here)."""
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(n=d, m=8)
    X, _ = synth.rank_one_samples(wl, seed=7, device="cuda", N=N)
    w = torch.rand(N, device="cuda", generator=torch.Generator("cuda").manual_seed(8)) * 3
    scale = 1.0 / (N * 5)
    with ffh.Handle(dtype="bf16") as h:
        C = h.weighted_gram(X, w, scale)
        C2 = h.weighted_gram(X, w, scale)
    torch.cuda.synchronize()
    assert torch.equal(C, C2), "the weighted Gram must be deterministic"
    Vn, wn = oracle.as_f64(X), oracle.as_f64(w)
    ref = oracle.weighted_gram(Vn, wn, scale)
    Cn = oracle.as_f64(C)
    assert np.array_equal(Cn, Cn.T), "output must be exactly symmetric"
    bound = _bf16_gram_bound(Vn, wn, scale) + 1e-7 * np.abs(ref).max()
    assert np.all(np.abs(Cn - ref) <= bound), np.max(np.abs(Cn - ref) / bound)
    # bf16 rounding of the weighted operand is unbiased (2^-9 relative per term, averaging
    # out over N terms); 5e-4 leaves a wide margin over the ~1e-4 measured
    rel = np.linalg.norm(Cn - ref) / np.linalg.norm(ref)
    assert rel < 5e-4, rel


def test_weighted_gram_f32_input():
    N, d = 2000, 100          # fp32 input: any d (internally padded to a multiple of 8)
    X = synth.gaussian(N, d, seed=3, device="cuda")
    w = torch.rand(N, device="cuda")
    with ffh.Handle(dtype="f32") as h:
        C = h.weighted_gram(X, w, 0.5)
    Vn, wn = oracle.as_f64(X), oracle.as_f64(w)
    ref = oracle.weighted_gram(Vn, wn, 0.5)
    # fp32 inputs are rounded to bf16 on both operands: 2 * 2^-9 + 2^-9
    bound = 3 * 2.0 ** -9 * 0.5 * ((np.abs(Vn).T * wn) @ np.abs(Vn)) + 1e-7 * np.abs(ref).max()
    assert np.all(np.abs(oracle.as_f64(C) - ref) <= bound)


# ---------------------------------------------------------------------------
# quadratic form
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N,d", [(1000, 64), (3000, 264), (1500, 512), (129, 1024), (700, 6400)])
def test_quad_form_matches_oracle(N, d):
    """d = 6400 has 25 column blocks of 256: four CTAs share each row block and their partial
    sums are added in a fixed order (the result must not depend on which CTA finishes first)."""
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(n=d, m=8)
    X, _ = synth.rank_one_samples(wl, seed=4, device="cuda", N=N)
    A = oracle.as_f64(synth.spd_matrix(d, seed=5, cond=1e3, dtype=torch.float64))
    Linv = oracle.tri_inverse(oracle.cholesky(A))
    with ffh.Handle(dtype="bf16") as h:
        Lt = torch.tensor(Linv, dtype=torch.float32, device="cuda")
        q = h.quad_form(X, Lt)
        q2 = h.quad_form(X, Lt)
    assert torch.equal(q, q2), "the quadratic form must be deterministic"
    Xn = oracle.as_f64(X)
    ref = oracle.inv_quad_forms_chol(oracle.cholesky(A), Xn)
    Lf = Linv.astype(np.float32).astype(np.float64)   # what the kernel is given
    y = Xn @ Lf.T
    z = np.abs(Xn) @ np.abs(Lf).T
    bound = (2.0 ** -8 * np.sum(np.abs(y) * z, 1) + 2.0 ** -18 * np.sum(z * z, 1)
             + 1e-5 * ref + np.abs(np.sum(y * y, 1) - ref))
    assert np.all(np.abs(oracle.as_f64(q) - ref) <= bound)


# ---------------------------------------------------------------------------
# Cholesky and inverse
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("d,cond", [(64, 1e2), (129, 1e2), (200, 1e3), (257, 1e3), (512, 1e3),
                                    (1000, 1e4), (1001, 1e3), (1536, 1e3), (2304, 1e3),
                                    (4096, 1e4), (8200, 1e3)])
def test_cholesky_matches_oracle(d, cond):
    """Cholesky factor L and inverse M = L^-1.  Unit roundoff of the arithmetic: bf16
    hi/lo split products on the tensor cores (u = 2^-16 per product, fp32 accumulation).
    Bounds: backward error ||L L^T - F|| / ||F|| <= 8 u_eff; inverse residual
    ||M L - I|| / sqrt(d) <= 8 u_eff sqrt(cond); forward error of L <= 8 u_eff cond;
    log|F| to d u_eff cond."""
    A = synth.spd_matrix(d, seed=6, cond=cond, dtype=torch.float32, device="cuda")
    with ffh.Handle() as h:
        L, Li, logdet = h.cholesky(A)
    An = oracle.as_f64(A)
    Lr = oracle.cholesky(An)
    Mr = oracle.tri_inverse(Lr)
    u_eff = 2.0 ** -16
    Ln, Mn = oracle.as_f64(L), oracle.as_f64(Li)
    assert np.all(np.triu(Ln, 1) == 0) and np.all(np.triu(Mn, 1) == 0)
    back = np.linalg.norm(Ln @ Ln.T - An) / np.linalg.norm(An)
    inv_res = np.linalg.norm(Mn @ Ln - np.eye(d)) / math.sqrt(d)
    eL = np.linalg.norm(Ln - Lr) / np.linalg.norm(Lr)
    eM = np.linalg.norm(Mn - Mr) / np.linalg.norm(Mr)
    print(f"d={d} cond={cond:g}: back={back:.2e} inv={inv_res:.2e} eL={eL:.2e} "
          f"eM={eM:.2e} dlogdet={abs(logdet - oracle.logdet_from_cholesky(Lr)):.2e}")
    assert back <= 8 * u_eff, back
    assert inv_res <= 8 * u_eff * math.sqrt(cond), inv_res
    assert eL <= 8 * u_eff * cond, eL
    assert eM <= 8 * u_eff * cond, eM
    assert abs(logdet - oracle.logdet_from_cholesky(Lr)) <= d * u_eff * cond


def test_cholesky_rejects_indefinite():
    A = torch.eye(300, device="cuda")
    A[150, 150] = -1.0
    with ffh.Handle() as h:
        with pytest.raises(ffh.FFHError) as ei:
            h.cholesky(A)
    assert ei.value.status == "FFH_ERR_NOT_SPD" and "150" in str(ei.value)


# ---------------------------------------------------------------------------
# the fit
# ---------------------------------------------------------------------------
FIT_CASES = {
    # the tiny rank-one configuration exactly (fp32, 10 iterations)
    "tiny_64": synth.WORKLOADS["tiny_64"],
    # bf16 LLM-like samples at a size the oracle finishes in seconds; m ragged vs 256
    "llama_small": synth.WORKLOADS["llama7b_attn_4096"].with_(N=16384, n=256, m=320, iters=4),
    # heavy-tailed inputs, n > m
    "student_small": synth.WORKLOADS["llama3_8b_down_14336x4096"].with_(N=20000, n=448, m=128,
                                                                        iters=4),
    # fp32 samples whose widths are not multiples of 8 (padded bf16 rows on the tensor path)
    "odd_f32": synth.WORKLOADS["tiny_64"].with_(N=3000, n=36, m=20, iters=5),
}


@pytest.mark.parametrize("case", sorted(FIT_CASES))
def test_fit_matches_oracle(case):
    wl = FIT_CASES[case]
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype=wl.dtype, final_loglik=True) as h:
        A, B = h.fit(X, G, iters=wl.iters)
        st = h.stats()
    ref = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=wl.iters)
    err = oracle.kron_rel_err(A.cpu(), B.cpu(), ref.A, ref.B)
    assert err <= 2e-3, err
    An = oracle.as_f64(A)
    assert np.trace(An) == pytest.approx(wl.n, rel=1e-4)
    assert np.array_equal(An, An.T)
    assert st["iters_done"] == wl.iters
    n, m = wl.n, wl.m
    # trace identity mean_k q_k r_k = m n after every half-step
    assert np.allclose(st["mean_qr"], m * n, rtol=2e-2)
    # log-likelihood: matches the oracle's trace and is non-decreasing
    ll = np.array(st["loglik"])
    assert np.allclose(ll, ref.loglik, rtol=1e-3, atol=1e-3 * np.abs(ref.loglik).max())


def test_fit_factorial_design_closed_form():
    """GPU fit of a factorial design reaches A (x) B = Sigma_x (x) Sigma_g."""
    # P = 4 n inputs and R = 4 m gradients keep Sigma_x, Sigma_g well conditioned (P = n
    # would make a square sample covariance, condition ~1e7, beyond any fp32 Cholesky)
    P, R, n, m = 1024, 512, 256, 128
    X, G, Xp, Gr = synth.factorial_design(P, R, n, m, seed=7, device="cuda", dtype=torch.bfloat16)
    Xp, Gr = oracle.as_f64(Xp), oracle.as_f64(Gr)
    Sx, Sg = Xp.T @ Xp / P, Gr.T @ Gr / R
    with ffh.Handle(dtype="bf16") as h:
        A, B = h.fit(X, G, iters=2)
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), Sx, Sg) <= 2e-3


def test_fit_host_inputs_equal_device_inputs():
    wl = FIT_CASES["llama_small"].with_(iters=2)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16") as h:
        A1, B1 = h.fit(X, G, iters=2)
        A2, B2 = h.fit(X.cpu().pin_memory(), G.cpu(), iters=2)
    assert torch.equal(A1.cpu(), A2) and torch.equal(B1.cpu(), B2)


def test_fit_damping_matches_oracle():
    wl = FIT_CASES["llama_small"].with_(iters=3)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16", damping=0.1) as h:
        A, B = h.fit(X, G, iters=3)
    ref = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=3, damping=0.1)
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), ref.A, ref.B) <= 2e-3


def test_fit_tol_stops_early():
    wl = FIT_CASES["tiny_64"]
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="f32") as h:
        h.fit(X, G, iters=50, tol=1e-4)
        st = h.stats()
    ref = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=50, tol=1e-4)
    assert st["iters_done"] < 50 and st["delta"] < 1e-4
    assert abs(st["iters_done"] - ref.iters_done) <= 1


@pytest.mark.parametrize("case,tol,final", [("tiny_64", 0.0, False), ("llama_small", 0.0, True),
                                             ("tiny_64", 1e-4, True)])
def test_fit_graph_replay_equals_direct_enqueue(case, tol, final):
    """A repeated fit on the same buffers replays the CUDA graph recorded by the first one;
    both must equal, bit for bit, the same fit enqueued kernel by kernel (no_graph), with
    the same statistics (a tol-stopped fit included) and the same kernel-launch count."""
    wl = FIT_CASES[case]
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    it = 40 if tol > 0 else wl.iters
    runs = {}
    for graph in (True, False):
        with ffh.Handle(dtype=wl.dtype, final_loglik=final, graph=graph) as h:
            out = []
            for _ in range(3):
                l0 = h.timings()["kernel_launches"]
                A, B = h.fit(X, G, iters=it, tol=tol)
                torch.cuda.synchronize()
                st = h.stats()
                out.append((A.cpu(), B.cpu(), st, h.timings()["kernel_launches"] - l0))
            runs[graph] = out
    A0, B0, st0, n0 = runs[False][0]
    labels = [f"graph fit {k}" for k in range(3)] + [f"direct fit {k}" for k in (1, 2)]
    for lab, (A, B, st, nl) in zip(labels, runs[True] + runs[False][1:]):
        assert torch.equal(A, A0) and torch.equal(B, B0), (
            lab, float((A - A0).norm() / A0.norm()), float((B - B0).norm() / B0.norm()))
        assert st["iters_done"] == st0["iters_done"]
        assert st["delta"] == st0["delta"] or (np.isnan(st["delta"]) and np.isnan(st0["delta"]))
        if final:
            assert np.array_equal(np.array(st["loglik"]), np.array(st0["loglik"]), equal_nan=True)
        assert nl == n0


def test_fit_graph_replay_keeps_profile_timings():
    """Profiling survives the replay: each replayed fit adds its Gram, quadratic-form and
    Cholesky intervals, as a directly enqueued fit does."""
    wl = FIT_CASES["llama_small"]
    X, G = synth.rank_one_samples(wl, seed=1, device="cuda")
    for graph in (True, False):
        with ffh.Handle(dtype="bf16", profile=True, graph=graph) as h:
            h.fit(X, G, iters=3)
            h.timings(reset=True)
            for _ in range(2):
                h.fit(X, G, iters=3)
            tm = h.timings()
        assert tm["gram_launches"] == 2 * 6 and tm["gram_ms"] > 0
        assert tm["qform_launches"] == 2 * 5 and tm["qform_ms"] > 0
        assert tm["chol_calls"] == 2 * 5 and tm["chol_ms"] > 0


@pytest.mark.parametrize("case,tol", [("tiny_64", 1e-4), ("llama_small", 2e-3)])
def test_stop_on_device_equals_fixed_count_fit(case, tol):
    """The stopping test runs on the device: the fit enqueues all `iters` iterations and
    the ones after delta_t < tol return at once.  The pair it returns, its statistics and
    its final log-likelihood must be bit-identical to a fit of exactly iters_done
    iterations (the fit is deterministic), and the skipped iterations must cost almost
    nothing."""
    wl = FIT_CASES[case]
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype=wl.dtype, final_loglik=True) as h:
        A1, B1 = h.fit(X, G, iters=60, tol=tol)
        st1 = h.stats()
        T = st1["iters_done"]
        assert 2 <= T < 60 and st1["delta"] < tol
        A2, B2 = h.fit(X, G, iters=T)
        st2 = h.stats()
        # timing: 60 enqueued iterations that stop at T against T iterations
        torch.cuda.synchronize()
        e = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
        e[0].record()
        h.fit(X, G, iters=60, tol=tol)
        e[1].record()
        e[2].record()
        h.fit(X, G, iters=T)
        e[3].record()
        torch.cuda.synchronize()
    assert torch.equal(A1, A2) and torch.equal(B1, B2)
    assert st2["iters_done"] == T
    assert np.array_equal(np.array(st1["loglik"]), np.array(st2["loglik"]))
    assert np.array_equal(np.array(st1["mean_qr"]), np.array(st2["mean_qr"]))
    assert math.isfinite(st1["loglik"][-1])
    t_stop, t_fixed = e[0].elapsed_time(e[1]), e[2].elapsed_time(e[3])
    print(f"\n{case}: stopped at {T} of 60; {t_stop:.2f} ms vs {t_fixed:.2f} ms for {T} iterations")
    # each skipped iteration is a few dozen launches that return at once
    assert t_stop < t_fixed + (60 - T) * 1.0 + 5.0


def test_stop_on_device_matrix_fit():
    wl = synth.WORKLOADS["kron_recovery_512x768"].with_(n=64, m=96)
    Gk = synth.matrix_samples(wl, seed=3, device="cuda", N=256)
    with ffh.Handle(dtype="f32", final_loglik=True) as h:
        A1, B1 = h.fit_matrix(Gk, 40, 1e-4)
        st1 = h.stats()
        T = st1["iters_done"]
        A2, B2 = h.fit_matrix(Gk, T, 0.0)
        st2 = h.stats()
    assert 2 <= T < 40
    assert torch.equal(A1, A2) and torch.equal(B1, B2)
    assert np.array_equal(np.array(st1["loglik"]), np.array(st2["loglik"]))
    ref = oracle.flipflop_fit_matrix(Gk.cpu(), iters=40, tol=1e-4)
    assert abs(T - ref.iters_done) <= 1


def test_fit_warm_start():
    wl = FIT_CASES["llama_small"].with_(iters=2)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    ref1 = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=1)
    ref3 = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=2, init_A=ref1.A)
    A0 = torch.tensor(ref1.A, dtype=torch.float32, device="cuda")
    with ffh.Handle(dtype="bf16", init_A=A0) as h:
        A, B = h.fit(X, G, iters=2)
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), ref3.A, ref3.B) <= 2e-3


# ---------------------------------------------------------------------------
# errors
# ---------------------------------------------------------------------------
def test_fit_argument_errors():
    X = torch.zeros(100, 16, dtype=torch.bfloat16, device="cuda")
    G = torch.zeros(100, 12, dtype=torch.bfloat16, device="cuda")
    with ffh.Handle(dtype="bf16") as h:
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X, G, iters=1)          # m = 12 is not a multiple of 8
        assert ei.value.status == "FFH_ERR_INVALID_ARG"
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X[:10], X[:10], iters=1)
        assert ei.value.status == "FFH_ERR_RANK"
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X, X, iters=0)
        assert ei.value.status == "FFH_ERR_INVALID_ARG"


def test_fault_injection_oom_and_pivot():
    wl = FIT_CASES["llama_small"].with_(iters=2)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16", fault=ffh.FAULT_OOM) as h:
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X, G, iters=2)
        assert ei.value.status == "FFH_ERR_OOM"
    with ffh.Handle(dtype="bf16", fault=ffh.FAULT_BAD_PIVOT) as h:
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X, G, iters=2)
        assert ei.value.status == "FFH_ERR_NOT_SPD"
    # the context is still usable afterwards
    with ffh.Handle(dtype="bf16") as h:
        A, B = h.fit(X, G, iters=1)
    assert torch.isfinite(A).all()


def test_fault_injection_lost_copy_times_out_and_context_survives():
    """FFH_FAULT_LOST_COPY: the Gram kernel's producer skips one staged copy, so the
    consumer's bounded wait (20 ms under fault injection) runs out.  The kernel must
    record FFH_ERR_TIMEOUT, drain what it issued, free its TMEM and return; the later
    kernels of the fit see the abort word and return at once; and the same context must
    then run a clean fit that matches the oracle."""
    wl = FIT_CASES["llama_small"].with_(iters=2)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16", fault=ffh.FAULT_LOST_COPY) as h:
        with pytest.raises(ffh.FFHError) as ei:
            h.fit(X, G, iters=2)
        assert ei.value.status == "FFH_ERR_TIMEOUT"
    torch.cuda.synchronize()
    with ffh.Handle(dtype="bf16") as h:
        A, B = h.fit(X, G, iters=2)
    ref = oracle.flipflop_fit(X.cpu(), G.cpu(), iters=2)
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), ref.A, ref.B) <= 2e-3


# ---------------------------------------------------------------------------
# matrix samples (Section 5, general G_k)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N,n,m,iters", [(256, 64, 96, 5), (300, 136, 72, 4), (96, 512, 768, 3)])
def test_fit_matrix_matches_oracle(N, n, m, iters):
    wl = synth.WORKLOADS["kron_recovery_512x768"].with_(n=n, m=m)
    Gk = synth.matrix_samples(wl, seed=3, device="cuda", N=N)
    with ffh.Handle(dtype="f32", final_loglik=True) as h:
        A, B = h.fit_matrix(Gk, iters=iters)
        st = h.stats()
    ref = oracle.flipflop_fit_matrix(Gk.cpu(), iters=iters)
    err = oracle.kron_rel_err(A.cpu(), B.cpu(), ref.A, ref.B)
    assert err <= 2e-3, err
    assert st["iters_done"] == iters
    assert np.allclose(st["mean_qr"], m * n, rtol=1e-6)
    assert np.allclose(st["loglik"], ref.loglik, rtol=1e-3, atol=1e-3 * np.abs(ref.loglik).max())


def test_fit_matrix_rank_one_samples_equal_rank_one_fit():
    """G_k = g_k x_k^T: the matrix-sample fit and the rank-one fit agree."""
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(N=2048, n=128, m=64, iters=3, dtype="f32")
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    Gk = torch.einsum("ki,kj->kij", G, X).contiguous()
    with ffh.Handle(dtype="f32") as h:
        A1, B1 = h.fit(X, G, iters=3)
        A2, B2 = h.fit_matrix(Gk, iters=3)
    assert oracle.kron_rel_err(A2.cpu(), B2.cpu(), A1.cpu(), B1.cpu()) <= 2e-3


def test_fit_matrix_host_input_and_damping():
    wl = synth.WORKLOADS["kron_recovery_512x768"].with_(n=64, m=48)
    Gk = synth.matrix_samples(wl, seed=4, device="cuda", N=200)
    with ffh.Handle(dtype="f32", damping=0.1) as h:
        A, B = h.fit_matrix(Gk.cpu(), iters=3)
    ref = oracle.flipflop_fit_matrix(Gk.cpu(), iters=3, damping=0.1)
    assert oracle.kron_rel_err(A, B, ref.A, ref.B) <= 2e-3


# ---------------------------------------------------------------------------
# Table 1 variants and the mismatch factor
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("case", ["tiny_64", "llama_small"])
def test_frobenius_fit_matches_oracle(case):
    wl = FIT_CASES[case].with_(iters=3)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype=wl.dtype, variant="frobenius") as h:
        A, B = h.fit(X, G, iters=wl.iters)
        st = h.stats()
    ref = oracle.frobenius_fit(X.cpu(), G.cpu(), iters=wl.iters)
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), ref.A, ref.B) <= 2e-3
    assert np.trace(oracle.as_f64(A)) == pytest.approx(wl.n, rel=1e-4)
    assert all(math.isnan(v) for v in st["loglik"])


@pytest.mark.parametrize("variant", ["input", "marginal"])
def test_input_and_marginal_hessians(variant):
    wl = FIT_CASES["llama_small"]
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    with ffh.Handle(dtype="bf16", variant=variant) as h:
        A, B = h.fit(X, G, iters=5)
        st = h.stats()
    if variant == "input":
        Ar, Br = oracle.input_hessian(X.cpu(), wl.m)
    else:
        Ar, Br = oracle.marginal_hessian(X.cpu(), G.cpu())
    assert oracle.kron_rel_err(A.cpu(), B.cpu(), Ar, Br) <= 2e-3
    assert st["iters_done"] == 1


def test_phi_tilde_matches_oracle_and_orders_variants():
    """Phi~ (Section 4 mismatch factor, sample form) of the four Table 1 Hessians: the
    GPU value matches the oracle's, and the FlipFlop fit has the smallest."""
    wl = FIT_CASES["llama_small"].with_(iters=6)
    X, G = synth.rank_one_samples(wl, seed=0, device="cuda")
    phis = {}
    for variant in ("flipflop", "frobenius", "input", "marginal"):
        with ffh.Handle(dtype="bf16", variant=variant) as h:
            A, B = h.fit(X, G, iters=wl.iters)
            phis[variant] = h.phi_tilde(X, G, A, B)
        ref = oracle.phi_tilde(X.cpu(), G.cpu(), A.cpu(), B.cpu())
        assert math.log(phis[variant]) == pytest.approx(math.log(ref), abs=2e-3), variant
    assert phis["flipflop"] <= min(phis["frobenius"], phis["input"], phis["marginal"]) * (1 + 1e-3)
