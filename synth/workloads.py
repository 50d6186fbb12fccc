"""Seeded synthetic calibration samples for the FlipFlop Hessian fit.

This module only draws inputs.  It holds none of the estimator's arithmetic and is
the one piece of code that both the fp64 oracle (``oracle/``) and the CUDA path's
tests and benchmark consume, so that both sides see the same bytes.

The paper fits A (x) B to calibration pairs (x_k, g_k) of one linear layer W in
R^{m x n}: x_k in R^n is the layer input and g_k in R^m the output gradient
(Section 5, problem statement; Appendix B, setup).  Its own calibration data
(Pile10k activations of Llama/Qwen layers) is not available here, so each named
workload below stands in for one layer shape with seeded Gaussian-type samples:

* power-law covariances  Sigma = Q diag(lambda) Q^T,  lambda_i = i^-p,  Q a
  seeded Haar-like orthogonal matrix (QR of a Gaussian matrix, signs fixed);
* "outlier channels": a seeded set of input features multiplied by a constant
  after the rotation (LLM activations have a few large channels);
* heavy tails: a multivariate Student-t with nu degrees of freedom,
  x = S z / sqrt(w / nu), w ~ chi^2_nu drawn as a sum of nu squared normals;
* matrix samples G_k = S_B Z_k S_A^T with S S^T = B0, A0 (Section 2 notation,
  M^{1/2} = S with S S^T = M), so that cov(vec G_k) = A0 (x) B0.

Everything is drawn with ``torch.Generator`` on the requested device in fixed-size
row chunks, so a given (workload, seed, device, N) always yields the same bytes.
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional

import torch

# rows drawn per chunk; fixed so that the bytes never depend on free memory
_CHUNK_ROWS = 16384

# independent random streams per tensor
_STREAM_QX, _STREAM_QG, _STREAM_ZX, _STREAM_ZG, _STREAM_OUT, _STREAM_W = range(6)
_STREAM_QA, _STREAM_QB, _STREAM_ZK = 10, 11, 12


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic layer shape.

    kind   "rank_one": samples (x_k, g_k), G_k = g_k x_k^T (Section 5);
           "matrix":   general matrix samples G_k in R^{m x n}.
    N      number of samples; n input features (A is n x n); m outputs (B is m x m).
    dtype  storage type of the samples, "f32" or "bf16".
    iters  flip-flop iterations of the fit (one iteration = B update then A update).
    """

    name: str
    kind: str
    N: int
    n: int
    m: int
    dtype: str
    iters: int
    x_exponent: float = 1.0
    g_exponent: float = 1.0
    x_outliers: int = 0
    outlier_scale: float = 1.0
    g_scale: float = 1.0
    student_nu: int = 0          # 0: Gaussian x; >0: multivariate Student-t x
    cond: float = 0.0            # matrix kind: condition number of A0 and B0

    def with_(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def torch_dtype(self) -> torch.dtype:
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    def sample_bytes(self) -> int:
        esize = 4 if self.dtype == "f32" else 2
        if self.kind == "matrix":
            return self.N * self.m * self.n * esize
        return self.N * (self.n + self.m) * esize


WORKLOADS = {
    # tiny rank-one fit, fp32, 10 iterations
    "tiny_64": Workload("tiny_64", "rank_one", N=4096, n=64, m=64, dtype="f32", iters=10),
    # Kronecker ground-truth recovery from matrix-normal samples, fp32, 20 iterations
    "kron_recovery_512x768": Workload(
        "kron_recovery_512x768", "matrix", N=65536, n=512, m=768, dtype="f32", iters=20,
        cond=1e3),
    # Llama-7B-like attention projection: 128 sequences x 2048 tokens
    "llama7b_attn_4096": Workload(
        "llama7b_attn_4096", "rank_one", N=262144, n=4096, m=4096, dtype="bf16", iters=8,
        x_outliers=8, outlier_scale=20.0, g_scale=1e-3),
    # Llama-7B-like MLP up projection
    "llama7b_mlp_up_4096x11008": Workload(
        "llama7b_mlp_up_4096x11008", "rank_one", N=262144, n=4096, m=11008, dtype="bf16",
        iters=8, x_outliers=8, outlier_scale=20.0, g_scale=1e-3),
    # Llama-3-8B-like down projection: 256 sequences x 2048 tokens, Student-t inputs
    "llama3_8b_down_14336x4096": Workload(
        "llama3_8b_down_14336x4096", "rank_one", N=524288, n=14336, m=4096, dtype="bf16",
        iters=8, student_nu=4, g_scale=1e-3),
}


def _gen(device, seed: int, stream: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed) * 1_000_003 + 7919 * stream + 17)
    return g


def power_law_spectrum(d: int, exponent: float) -> torch.Tensor:
    """lambda_i = i^-exponent, i = 1..d (fp64, host)."""
    i = torch.arange(1, d + 1, dtype=torch.float64)
    return i.pow(-exponent)


def exponent_for_condition(d: int, cond: float) -> float:
    """Power-law exponent p with lambda_1 / lambda_d = d^p = cond."""
    return math.log(cond) / math.log(d) if d > 1 else 0.0


_ORTHO_CACHE: dict = {}


def orthogonal(d: int, gen: torch.Generator, device) -> torch.Tensor:
    """Seeded orthogonal d x d matrix (fp32): QR of a Gaussian matrix, signs fixed.

    The Gaussian matrix is drawn on the generator's device; the QR runs on the host in
    fp64 (no device linear-algebra library is needed to draw inputs).  A generator that
    has drawn nothing yet always gives the same matrix, so those results are kept (the
    large host QRs are then done once per process)."""
    fresh = torch.Generator(device=gen.device)
    fresh.manual_seed(gen.initial_seed())
    key = (d, str(torch.device(device)), gen.initial_seed())
    if torch.equal(gen.get_state(), fresh.get_state()) and key in _ORTHO_CACHE:
        torch.randn(d, d, generator=gen, device=device, dtype=torch.float32)  # same draw
        return _ORTHO_CACHE[key].to(device)
    was_fresh = torch.equal(gen.get_state(), fresh.get_state())
    a = torch.randn(d, d, generator=gen, device=device, dtype=torch.float32)
    q, r = torch.linalg.qr(a.to("cpu", torch.float64))
    s = torch.sign(torch.diagonal(r))
    s[s == 0] = 1
    out = (q * s.unsqueeze(0)).to(torch.float32)
    if was_fresh and d >= 1024:
        _ORTHO_CACHE[key] = out
    return out.to(device=device)


def sqrt_cov(d: int, exponent: float, gen: torch.Generator, device) -> torch.Tensor:
    """S = Q diag(lambda)^{1/2} (fp32), so S S^T = Q diag(lambda) Q^T."""
    q = orthogonal(d, gen, device)
    lam = power_law_spectrum(d, exponent).to(device=device, dtype=torch.float32)
    return q * lam.sqrt().unsqueeze(0)


def _rows(N: int):
    for r0 in range(0, N, _CHUNK_ROWS):
        yield r0, min(N, r0 + _CHUNK_ROWS)


def rank_one_samples(wl: Workload, seed: int = 0, device="cpu", N: Optional[int] = None):
    """Return (X, G): X is N x n, G is N x m, row k = x_k^T, g_k^T, dtype wl.dtype.

    x_k = S_x z_k (Gaussian) or S_x z_k / sqrt(w_k / nu) (Student-t), then the
    outlier channels are scaled; g_k = g_scale * S_g z'_k.
    """
    assert wl.kind == "rank_one"
    N = wl.N if N is None else int(N)
    dev = torch.device(device)
    Sx = sqrt_cov(wl.n, wl.x_exponent, _gen(dev, seed, _STREAM_QX), dev)
    Sg = sqrt_cov(wl.m, wl.g_exponent, _gen(dev, seed, _STREAM_QG), dev)
    col_scale = torch.ones(wl.n, device=dev, dtype=torch.float32)
    if wl.x_outliers:
        go = _gen(dev, seed, _STREAM_OUT)
        idx = torch.randperm(wl.n, generator=go, device=dev)[: wl.x_outliers]
        col_scale[idx] = wl.outlier_scale
    X = torch.empty(N, wl.n, device=dev, dtype=wl.torch_dtype)
    G = torch.empty(N, wl.m, device=dev, dtype=wl.torch_dtype)
    gzx, gzg, gw = (_gen(dev, seed, s) for s in (_STREAM_ZX, _STREAM_ZG, _STREAM_W))
    SxT, SgT = Sx.t().contiguous(), Sg.t().contiguous()
    for r0, r1 in _rows(N):
        z = torch.randn(r1 - r0, wl.n, generator=gzx, device=dev, dtype=torch.float32)
        x = z @ SxT
        if wl.student_nu:
            w = torch.randn(r1 - r0, wl.student_nu, generator=gw, device=dev,
                            dtype=torch.float32).square().sum(1)
            x = x * torch.rsqrt(w / wl.student_nu).unsqueeze(1)
        x = x * col_scale
        X[r0:r1] = x.to(wl.torch_dtype)
        zg = torch.randn(r1 - r0, wl.m, generator=gzg, device=dev, dtype=torch.float32)
        G[r0:r1] = (zg @ SgT * wl.g_scale).to(wl.torch_dtype)
    return X, G


def matrix_normal_factors(wl: Workload, seed: int = 0, device="cpu"):
    """Return (S_A, S_B, A0, B0) for the matrix workload: A0 = S_A S_A^T (n x n),
    B0 = S_B S_B^T (m x m), power-law spectra with condition number wl.cond."""
    dev = torch.device(device)
    pa = exponent_for_condition(wl.n, wl.cond)
    pb = exponent_for_condition(wl.m, wl.cond)
    SA = sqrt_cov(wl.n, pa, _gen(dev, seed, _STREAM_QA), dev)
    SB = sqrt_cov(wl.m, pb, _gen(dev, seed, _STREAM_QB), dev)
    return SA, SB, SA @ SA.t(), SB @ SB.t()


def matrix_samples(wl: Workload, seed: int = 0, device="cpu", N: Optional[int] = None,
                   out: Optional[torch.Tensor] = None):
    """Return Gk, an N x m x n tensor (row-major per sample) with
    G_k = S_B Z_k S_A^T, Z_k iid N(0,1)."""
    assert wl.kind == "matrix"
    N = wl.N if N is None else int(N)
    dev = torch.device(device)
    SA, SB, _, _ = matrix_normal_factors(wl, seed, dev)
    Gk = out if out is not None else torch.empty(N, wl.m, wl.n, device=dev,
                                                  dtype=wl.torch_dtype)
    gz = _gen(dev, seed, _STREAM_ZK)
    chunk = max(1, _CHUNK_ROWS // 64)
    SAT = SA.t().contiguous()
    for k0 in range(0, N, chunk):
        k1 = min(N, k0 + chunk)
        z = torch.randn(k1 - k0, wl.m, wl.n, generator=gz, device=dev, dtype=torch.float32)
        Gk[k0:k1] = torch.matmul(torch.matmul(SB, z), SAT).to(Gk.dtype)
    return Gk


def rademacher(N: int, d: int, seed: int = 0, device="cpu", dtype=torch.float32):
    """N x d matrix of independent +-1 entries."""
    g = _gen(torch.device(device), seed, 99)
    b = torch.randint(0, 2, (N, d), generator=g, device=device)
    return (2 * b - 1).to(dtype)


def gaussian(N: int, d: int, seed: int = 0, stream: int = 0, device="cpu",
             dtype=torch.float32, scale: float = 1.0):
    """N x d iid N(0, scale^2) matrix."""
    g = _gen(torch.device(device), seed, 200 + stream)
    return (torch.randn(N, d, generator=g, device=device, dtype=torch.float32) * scale).to(dtype)


def factorial_design(P: int, R: int, n: int, m: int, seed: int = 0, device="cpu",
                     dtype=torch.float32):
    """All N = P*R pairs of P input vectors and R gradient vectors.

    Returns (X, G, Xp, Gr): X, G are the N x n / N x m sample matrices (sample
    k = p*R + r pairs x_p with g_r); Xp (P x n) and Gr (R x m) are the distinct
    vectors.  For this design H = E[x x^T] (x) E[g g^T] holds exactly.
    """
    dev = torch.device(device)
    Sx = sqrt_cov(n, 1.0, _gen(dev, seed, 300), dev)
    Sg = sqrt_cov(m, 1.0, _gen(dev, seed, 301), dev)
    Xp = torch.randn(P, n, generator=_gen(dev, seed, 302), device=dev) @ Sx.t()
    Gr = torch.randn(R, m, generator=_gen(dev, seed, 303), device=dev) @ Sg.t()
    Xp, Gr = Xp.to(dtype), Gr.to(dtype)
    X = Xp.repeat_interleave(R, dim=0)
    G = Gr.repeat(P, 1)
    return X.contiguous(), G.contiguous(), Xp, Gr


def spd_matrix(d: int, seed: int = 0, cond: float = 100.0, device="cpu",
               dtype=torch.float32, stream: int = 400) -> torch.Tensor:
    """Seeded SPD matrix Q diag(lambda) Q^T with a power-law spectrum of the given
    condition number (used as a seeded input to single steps of the fit)."""
    dev = torch.device(device)
    p = exponent_for_condition(d, cond)
    S = sqrt_cov(d, p, _gen(dev, seed, stream), dev).to(torch.float64)
    A = S @ S.t()
    A = 0.5 * (A + A.t())
    return A.to(dtype)
