"""ffh_weighted_gram_static: the weighted Gram for callers that cannot allocate device
memory (their framework owns every byte of it, or an allocation would stall a
latency-critical path).  Its working memory is a fixed static device array, so it
must give the same Gram as ffh_weighted_gram, call after call, even though the array
keeps the previous call's contents.  This file is collected last on purpose."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_14706_gb300 as ffh
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_14706_gb300 import build
    build.build()
    return ffh.load_library()


def _call_static(lib, V, w, scale):
    N, d = V.shape
    C = torch.empty(d, d, dtype=torch.float32, device="cuda")
    buf = ctypes.create_string_buffer(256)
    code = lib.ffh_weighted_gram_static(
        ctypes.c_void_p(V.data_ptr()), None if w is None else ctypes.c_void_p(w.data_ptr()),
        N, d, scale, ctypes.c_void_p(C.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream), buf, 256)
    return code, C, buf.value.decode()


def _bound(V, w, scale):
    # the tolerance of the Gram parity tests: one bf16 rounding of the weighted operand
    Va = np.abs(oracle.as_f64(V))
    wa = np.ones(V.shape[0]) if w is None else np.abs(oracle.as_f64(w))
    return 2.0 ** -8 * scale * ((Va.T * wa) @ Va)


def test_static_gram_matches_allocating_entry_point_twice(lib):
    wl = synth.WORKLOADS["llama7b_attn_4096"].with_(n=384, m=8)
    X, _ = synth.rank_one_samples(wl, seed=11, device="cuda", N=9000)
    g = torch.Generator("cuda").manual_seed(5)
    w1 = torch.rand(9000, device="cuda", generator=g) * 2
    # second call: fewer samples, so stale weights of the first call beyond N would show
    X2 = X[:5001].contiguous()
    w2 = torch.rand(5001, device="cuda", generator=g)
    with ffh.Handle(dtype="bf16") as h:
        ref1 = h.weighted_gram(X, w1, 1e-3)
        ref2 = h.weighted_gram(X2, w2, 2e-3)
    for V, w, scale, ref in ((X, w1, 1e-3, ref1), (X2, w2, 2e-3, ref2)):
        code, C, msg = _call_static(lib, V, w, scale)
        assert code == 0, msg
        torch.cuda.synchronize()
        Cn = oracle.as_f64(C)
        # against the oracle's weighted Gram directly, then against the allocating entry
        exact = oracle.weighted_gram(oracle.as_f64(V), oracle.as_f64(w), scale)
        bound = _bound(V, w, scale) + 1e-7 * np.abs(exact).max()
        assert np.all(np.abs(Cn - exact) <= bound), np.max(np.abs(Cn - exact) / bound)
        assert np.all(np.abs(Cn - oracle.as_f64(ref)) <= 2 * bound)
        assert np.array_equal(Cn, Cn.T)


def test_static_gram_unweighted_and_rejects_oversize(lib):
    X = synth.gaussian(3000, 64, seed=12, device="cuda", dtype=torch.bfloat16)
    with ffh.Handle(dtype="bf16") as h:
        ref = h.weighted_gram(X, None, 0.5)
    code, C, msg = _call_static(lib, X, None, 0.5)
    assert code == 0, msg
    Cn = oracle.as_f64(C)
    exact = oracle.weighted_gram(oracle.as_f64(X), np.ones(X.shape[0]), 0.5)
    assert np.all(np.abs(Cn - exact) <= _bound(X, None, 0.5) + 1e-7)
    assert np.all(np.abs(Cn - oracle.as_f64(ref)) <= 2 * _bound(X, None, 0.5) + 1e-7)
    big = torch.empty(64, 8192, dtype=torch.bfloat16, device="cuda")
    code, _, msg = _call_static(lib, big, None, 1.0)
    assert code == 1 and "static scratch" in msg
