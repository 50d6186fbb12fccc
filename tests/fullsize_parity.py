#!/usr/bin/env python
"""Full-size parity of the CUDA FlipFlop fit against the fp64 oracle.

The five benchmark configurations are too large for an oracle fit inside the GPU test run
(the fp64 fit of the 14336 x 4096 layer takes hours of host time), so the comparison
runs in two halves that share only the portable seeded inputs (``synth.portable``):

  gpu     on a GPU machine: draw each configuration's samples, fit them with the CUDA
          library (libffh, through the C ABI), and save for each trace-normalised
          factor F^ = F / tr F its squared norm, its diagonal and the sketch F^ Omega
          (Omega a seeded d x k Gaussian matrix), plus the full factors when they are
          small; also the sha256 of the samples.
  oracle  on any host: draw the same samples, check the sha256, run the oracle fit
          (cached on disk by input digest and oracle source digest) and compare.

With E = F^ - F^' (GPU minus oracle), ||E Omega||_F^2 / k is an unbiased estimate of
||E||_F^2 (E[Omega Omega^T] = k I), with relative spread about sqrt(2 / (k r)) for an
error of effective rank r; the per-column terms give its standard error.  From the
exact squared norms of both factors and the estimated ||E||^2,
<F^, F^'> = (||F^||^2 + ||F^'||^2 - ||E||^2) / 2, and the relative Frobenius error
of the trace-normalised A (x) B follows in closed form:
  err^2 = (|A^|^2 |B^|^2 + |A^'|^2 |B^'|^2 - 2 <A^,A^'> <B^,B^'>) / (|A^'|^2 |B^'|^2).

  python tests/fullsize_parity.py gpu    --out DIR [--configs a,b,...]
  python tests/fullsize_parity.py oracle --gpu DIR [--configs a,b,...] [--cache DIR]
  python tests/fullsize_parity.py oracle --fit-only [--configs a,b,...]
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

import synth  # noqa: E402
from synth import portable  # noqa: E402

ALL = ["tiny_64", "kron_recovery_512x768", "llama7b_attn_4096", "llama7b_mlp_up_4096x11008",
       "llama3_8b_down_14336x4096"]
SKETCH_K = 64
FULL_MAX_D = 1024      # factors up to this size are saved whole
SEED = 0


def omega(d: int, k: int = SKETCH_K) -> np.ndarray:
    """Seeded d x k Gaussian test matrix (the same on every machine)."""
    g = np.random.Generator(np.random.PCG64(np.random.SeedSequence([SEED, 7777, d, k])))
    return g.standard_normal((d, k))


def factor_summary(F: np.ndarray) -> dict:
    Fh = F / np.trace(F)
    out = {"norm2": float(np.sum(Fh * Fh)), "diag": np.diag(Fh).copy(),
           "sketch": Fh @ omega(F.shape[0])}
    if F.shape[0] <= FULL_MAX_D:
        out["full"] = Fh
    return out


# ---------------------------------------------------------------------------
# GPU half
# ---------------------------------------------------------------------------
def run_gpu(args) -> int:
    import paper_2609_14706_gb300 as ffh

    os.makedirs(args.out, exist_ok=True)
    torch.cuda.set_device(0)
    for name in args.configs:
        wl = synth.WORKLOADS[name]
        t0 = time.time()
        matrix = wl.kind == "matrix"
        if matrix:
            Gk = portable.matrix_samples(wl, seed=SEED, device="cuda")
            data = (Gk,)
        else:
            X, G = portable.rank_one_samples(wl, seed=SEED, device="cuda")
            data = (X, G)
        torch.cuda.synchronize()
        t_gen = time.time() - t0
        digest = portable.sha256(*data)

        def fit(h):
            if matrix:
                return h.fit_matrix(Gk, wl.iters)
            return h.fit(X, G, iters=wl.iters)

        with ffh.Handle(dtype=wl.dtype) as h:
            A, B = fit(h)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            A, B = fit(h)
            e1.record()
            torch.cuda.synchronize()
            stats = h.stats()
        An = A.double().cpu().numpy()
        Bn = B.double().cpu().numpy()
        sa, sb = factor_summary(An), factor_summary(Bn)
        rec = {"workload": name, "sha256": digest, "N": wl.N, "n": wl.n, "m": wl.m,
               "iters": wl.iters, "fit_ms": e0.elapsed_time(e1), "gen_s": t_gen,
               "loglik": [float(v) for v in stats["loglik"]],
               "mean_qr": [float(v) for v in stats["mean_qr"]]}
        arrays = {}
        for tag, s in (("A", sa), ("B", sb)):
            for key, val in s.items():
                if key == "norm2":
                    rec[f"{tag}_norm2"] = val
                else:
                    arrays[f"{tag}_{key}"] = val
        np.savez_compressed(os.path.join(args.out, f"{name}.npz"), **arrays)
        with open(os.path.join(args.out, f"{name}.json"), "w") as f:
            json.dump(rec, f)
        print(json.dumps({k: v for k, v in rec.items() if k not in ("loglik", "mean_qr")}),
              flush=True)
        del data, A, B
        X = G = Gk = None
        torch.cuda.empty_cache()
    return 0


# ---------------------------------------------------------------------------
# oracle half
# ---------------------------------------------------------------------------
def oracle_source_digest() -> str:
    with open(os.path.join(ROOT, "oracle", "flipflop.py"), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def oracle_fit_cached(name: str, wl, X, G, digest: str, cache: str, tol: float = 0.0,
                      blocks=None):
    """The oracle fit of the workload (all wl.iters iterations, or until delta_t < tol:
    past the fixed point further iterations move the factors by less than tol)."""
    import oracle

    os.makedirs(cache, exist_ok=True)
    tag = "" if tol == 0.0 else f"_tol{tol:g}"
    path = os.path.join(cache, f"{name}_{digest[:16]}_{oracle_source_digest()[:12]}{tag}.npz")
    if os.path.exists(path):
        z = np.load(path)
        return z["A"], z["B"], float(z["seconds"]), json.loads(str(z["deltas"]))
    t0 = time.time()

    def progress(t, delta):
        print(f"  [{name}] oracle iteration {t}/{wl.iters} done at {time.time() - t0:.0f} s "
              f"(delta {delta:.3e})", flush=True)

    if blocks is not None:
        A, B, _, dl = oracle.flipflop_fit_matrix_blocks(blocks, wl.N, wl.m, wl.n, wl.iters,
                                                        tol=tol, progress=progress)
    else:
        fit = oracle.flipflop_fit(X, G, iters=wl.iters, tol=tol, progress=progress)
        A, B, dl = fit.A, fit.B, fit.deltas
    sec = time.time() - t0
    deltas = [None if math.isinf(d) else d for d in dl]
    np.savez(path, A=A, B=B, seconds=sec, deltas=json.dumps(deltas))
    return A, B, sec, deltas


def sketch_err2(sketch_gpu: np.ndarray, F_ref: np.ndarray):
    """(estimate of ||F^_gpu - F^_ref||_F^2, its standard error) from the sketches."""
    R = (F_ref / np.trace(F_ref)) @ omega(F_ref.shape[0])
    cols = np.sum((sketch_gpu - R) ** 2, axis=0)        # ||E omega_j||^2, mean ||E||^2
    return float(np.mean(cols)), float(np.std(cols, ddof=1) / math.sqrt(cols.size))


def compare(rec: dict, arr, A_ref: np.ndarray, B_ref: np.ndarray) -> dict:
    a2, b2 = rec["A_norm2"], rec["B_norm2"]
    Ah, Bh = A_ref / np.trace(A_ref), B_ref / np.trace(B_ref)
    a2r, b2r = float(np.sum(Ah * Ah)), float(np.sum(Bh * Bh))
    out = {}
    if "A_full" in arr and "B_full" in arr:
        eA2 = float(np.sum((arr["A_full"] - Ah) ** 2))
        eB2 = float(np.sum((arr["B_full"] - Bh) ** 2))
        seA = seB = 0.0
        out["method"] = "exact (full factors)"
    else:
        eA2, seA = sketch_err2(arr["A_sketch"], A_ref)
        eB2, seB = sketch_err2(arr["B_sketch"], B_ref)
        out["method"] = f"sketch k={SKETCH_K}"

    def kron_err(ea2, eb2):
        ipa = (a2 + a2r - ea2) / 2.0
        ipb = (b2 + b2r - eb2) / 2.0
        num = a2 * b2 + a2r * b2r - 2.0 * ipa * ipb
        return math.sqrt(max(num, 0.0) / (a2r * b2r))

    err = kron_err(eA2, eB2)
    hi = kron_err(eA2 + 2 * seA, eB2 + 2 * seB)
    out.update({
        "kron_rel_err": err, "kron_rel_err_2se_upper": hi,
        "A_rel_err": math.sqrt(eA2 / a2r), "B_rel_err": math.sqrt(eB2 / b2r),
        "A_diag_max_rel": float(np.max(np.abs(arr["A_diag"] - np.diag(Ah)) / np.abs(np.diag(Ah)))),
        "B_diag_max_rel": float(np.max(np.abs(arr["B_diag"] - np.diag(Bh)) / np.abs(np.diag(Bh)))),
        "A_norm_rel": abs(math.sqrt(a2) - math.sqrt(a2r)) / math.sqrt(a2r),
        "B_norm_rel": abs(math.sqrt(b2) - math.sqrt(b2r)) / math.sqrt(b2r),
    })
    return out


def run_oracle(args) -> int:
    status = 0
    for name in args.configs:
        wl = synth.WORKLOADS[name]
        t0 = time.time()
        blocks = None
        if wl.kind == "matrix":
            # 103 GB of samples at the full size: drawn block by block on every pass
            X = G = None

            def blocks(wl=wl):
                for _, blk in portable.matrix_blocks(wl, seed=SEED, device="cpu"):
                    yield blk

            hsh = hashlib.sha256()
            for blk in blocks():
                hsh.update(blk.contiguous().view(-1).view(torch.uint8).numpy().tobytes())
            digest = hsh.hexdigest()
        else:
            X, G = portable.rank_one_samples(wl, seed=SEED, device="cpu")
            digest = portable.sha256(X, G)
        t_gen = time.time() - t0
        tol = args.oracle_tol if name in args.tol_configs else 0.0
        if args.fit_only:
            _, _, sec, _ = oracle_fit_cached(name, wl, X, G, digest, args.cache, tol, blocks)
            print(json.dumps({"workload": name, "sha256": digest, "oracle_fit_s": sec,
                              "host_gen_s": t_gen}), flush=True)
            del X, G
            continue
        with open(os.path.join(args.gpu, f"{name}.json")) as f:
            rec = json.load(f)
        arr = dict(np.load(os.path.join(args.gpu, f"{name}.npz")))
        if digest != rec["sha256"]:
            print(json.dumps({"workload": name, "error": "input digests differ",
                              "gpu": rec["sha256"], "host": digest}), flush=True)
            status = 1
            continue
        A_ref, B_ref, sec, deltas = oracle_fit_cached(name, wl, X, G, digest, args.cache, tol,
                                                      blocks)
        cmp = compare(rec, arr, A_ref, B_ref)
        line = {"workload": name, "N": wl.N, "n": wl.n, "m": wl.m, "iters": wl.iters,
                "dtype": wl.dtype, "sha256": digest, **cmp,
                "gpu_fit_ms": rec["fit_ms"], "oracle_fit_s": sec,
                "oracle_iters": len(deltas), "oracle_last_delta": deltas[-1],
                "oracle_cores": len(os.sched_getaffinity(0)), "host_gen_s": t_gen,
                "tolerance": 2e-3, "pass": cmp["kron_rel_err_2se_upper"] <= 2e-3}
        print(json.dumps(line), flush=True)
        if not line["pass"]:
            status = 1
        del X, G
    return status


def main() -> int:
    p = argparse.ArgumentParser()
    p.add_argument("half", choices=["gpu", "oracle"])
    p.add_argument("--configs", default=",".join(ALL))
    p.add_argument("--out", default=os.path.join(ROOT, "parity_out"))
    p.add_argument("--gpu", default=os.path.join(ROOT, "parity_out"))
    p.add_argument("--cache", default=os.path.join(ROOT, "tests", ".oracle_cache"))
    p.add_argument("--oracle-tol", type=float, default=1e-12,
                   help="oracle stopping tolerance for the --tol-configs workloads")
    p.add_argument("--tol-configs", default="llama3_8b_down_14336x4096,kron_recovery_512x768",
                   help="workloads whose oracle fit stops at --oracle-tol (the rest run "
                        "all their iterations)")
    p.add_argument("--fit-only", action="store_true",
                   help="oracle half: only run (and cache) the oracle fits")
    args = p.parse_args()
    args.configs = [c for c in args.configs.split(",") if c]
    args.tol_configs = [c for c in args.tol_configs.split(",") if c]
    return run_gpu(args) if args.half == "gpu" else run_oracle(args)


if __name__ == "__main__":
    sys.exit(main())
