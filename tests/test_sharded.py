"""Sample-sharded fit: the driver's reduction over ranks, run as gloo processes on the CPU.

Each rank holds a disjoint shard of the samples; the steps are the oracle's (fp64, CPU),
so the only thing under test is the driver: the order of the half-steps, the sum over
ranks of the unscaled partial Grams, the MLE scales with the total sample count, the
damping, the tr(A) = n rescale and the stopping statistic.  The sharded fit must equal
the single-process oracle fit of all samples (Section 5: each update is a sum over the
samples, so splitting the sum changes only the order of the additions)."""
import math
import os
import socket

import numpy as np
import pytest
import torch

import oracle

N, n, m = 1001, 6, 5      # ragged: 1001 samples over 2 ranks / 3 shards


def _samples(seed=0):
    rng = np.random.default_rng(seed)
    Sx = rng.standard_normal((n, n)) / math.sqrt(n) + np.eye(n)
    Sg = rng.standard_normal((m, m)) / math.sqrt(m) + np.eye(m)
    X = rng.standard_normal((N, n)) @ Sx.T
    G = rng.standard_normal((N, m)) @ Sg.T * (1.0 + 0.5 * np.abs(X[:, :1]))
    return X, G


class OracleSteps:
    """The four steps of a sharded half-step with the oracle's fp64 arithmetic."""

    def __init__(self, damping: float):
        self.lam = damping

    def partial_gram(self, shards, F):
        L = None if F is None else oracle.cholesky(F.numpy())
        P = None
        for U, V in shards:
            Un, Vn = oracle.as_f64(U), oracle.as_f64(V)
            w = np.einsum("kd,kd->k", Un, Un) if L is None else oracle.inv_quad_forms_chol(L, Un)
            Pi = oracle.weighted_gram(Vn, w, 1.0)
            P = Pi if P is None else P + Pi
        return torch.from_numpy(P)

    def update_from_sum(self, P, scale):
        return torch.from_numpy(oracle.damp(scale * P.numpy(), self.lam))

    def normalize_pair(self, A, B):
        s = float(torch.trace(A)) / A.shape[0]
        A /= s
        B *= s
        return s

    def relative_change(self, F, Fprev):
        return oracle.rel_change(F.numpy(), Fprev.numpy())


def _worker(rank, world, port, iters, tol, damping, out):
    import torch.distributed as dist

    from paper_2609_14706_gb300.sharded import fit_sharded

    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        X, G = _samples()
        Xt, Gt = torch.from_numpy(X), torch.from_numpy(G)
        if rank == 0:   # two shards in this process: rows 0..299 and 300..499
            shards = [(Xt[:300], Gt[:300]), (Xt[300:500], Gt[300:500])]
        else:           # one shard: rows 500..1000
            shards = [(Xt[500:], Gt[500:])]
        res = fit_sharded(shards, iters, tol=tol, reduce_sum=dist.all_reduce,
                          steps=OracleSteps(damping))
        out.put((rank, res.A.numpy(), res.B.numpy(), res.deltas, res.iters_done))
    finally:
        dist.destroy_process_group()


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run(iters, tol, damping):
    ctx = torch.multiprocessing.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, iters, tol, damping, out))
             for r in range(2)]
    for p in procs:
        p.start()
    res = {}
    for _ in procs:
        rank, A, B, deltas, t = out.get(timeout=300)
        res[rank] = (A, B, deltas, t)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return res


@pytest.mark.parametrize("iters,tol,damping", [(6, 0.0, 0.0), (60, 1e-9, 0.0), (5, 0.0, 0.1)])
def test_sharded_fit_equals_single_process_fit(iters, tol, damping):
    res = _run(iters, tol, damping)
    X, G = _samples()
    ref = oracle.flipflop_fit(X, G, iters=iters, tol=tol, damping=damping)
    for rank in (0, 1):
        A, B, deltas, t = res[rank]
        assert t == ref.iters_done
        ea, eb = oracle.factor_rel_errs(A, B, ref.A, ref.B)
        assert ea < 1e-12 and eb < 1e-12, (ea, eb)
        assert np.trace(A) == pytest.approx(n, rel=1e-13)
        assert math.isinf(deltas[0])
        assert np.allclose(deltas[1:], ref.deltas[1:], rtol=1e-6, atol=1e-14)
    # every rank holds the same factors (the sum over ranks is the same everywhere)
    assert np.array_equal(res[0][0], res[1][0]) and np.array_equal(res[0][1], res[1][1])
