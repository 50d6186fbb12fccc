"""Portable seeded samples: the same bytes on any host and on any device.

The default generators (``workloads.py``) draw with torch's device generators, whose
streams differ between the CPU and a GPU.  The full-size parity runs need the fp64
oracle (on one machine's host cores) and the CUDA fit (on a GPU machine) to see the
same samples, so this module draws them in a way that does not depend on the machine:

* every normal variate comes from numpy's PCG64 generator (integer state), seeded by a
  SeedSequence of (seed, stream[, chunk]), in fp64, one generator per fixed chunk of
  rows, so the bytes do not depend on how many threads draw them;
* the mixing x = S z is exact in fp64: z is put on a grid of 2^-8 (clipped to |z| <= 8)
  and S on a grid of 2^-26 (|S_ij| <= 1), so every product is an integer multiple of
  2^-34 below 2^37 of those units and every partial sum of up to 2^14 of them stays
  below 2^51 < 2^53: any order of the additions (another BLAS, a GPU) gives the same
  result, bit for bit;
* the remaining steps (the Student-t factor, outlier and g scales) are single IEEE
  operations per element, and the result is rounded once to fp32 and then, for bf16
  workloads, to bf16 (both round-to-nearest-even).

The grids are far finer than anything the statistics of a fit can see (the normal
variate moves by at most 2^-9, an entry of S by 2^-27).  ``sha256`` digests the bytes so
that both sides can confirm they saw the same samples.

The recipe is the one of ``workloads.py`` (power-law covariances with a Haar-like
rotation, outlier channels, multivariate Student-t inputs, g scale); only the random
streams differ.  This module holds none of the estimator's arithmetic.
"""
from __future__ import annotations

import hashlib
import os
from concurrent.futures import ThreadPoolExecutor
from typing import Optional

import numpy as np
import torch

from .workloads import Workload, exponent_for_condition

# rows per generator chunk; fixed, so the bytes never depend on memory or threads
CHUNK_ROWS = 8192
# the exact-mixing grids: z in 2^-Z_BITS units (|z| <= Z_CLIP), S in 2^-S_BITS units
Z_BITS, Z_CLIP, S_BITS = 8, 8.0, 26
# matrix samples: the intermediate S_B Z_k is put on a 2^-Y_BITS grid (|.| <= Y_CLIP) and
# S_A on a 2^-SA_BITS grid, so the second product is exact as well (512 terms)
Y_BITS, Y_CLIP, SA_BITS = 12, 1024.0, 20

# stream keys (a namespace of their own: 1000 + k)
_QX, _QG, _ZX, _ZG, _OUT, _W, _QA, _QB, _ZK = (1000 + k for k in range(9))


def _rng(seed: int, *key: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), *map(int, key)])))


def orthogonal64(d: int, seed: int, stream: int) -> np.ndarray:
    """Seeded orthogonal d x d matrix (fp64): QR of a Gaussian matrix, signs fixed so
    that R has a positive diagonal (a Haar-distributed rotation)."""
    a = _rng(seed, stream).standard_normal((d, d))
    q, r = np.linalg.qr(a)
    s = np.sign(np.diag(r))
    s[s == 0] = 1.0
    return q * s[None, :]


def _grid(a: np.ndarray, bits: int, clip: float = None) -> np.ndarray:
    """Nearest multiple of 2^-bits (ties to even; exact in fp64 for |a| < 2^(53 - bits))."""
    if clip is not None:
        a = np.clip(a, -clip, clip)
    return np.rint(a * (2.0 ** bits)) * (2.0 ** -bits)


def sqrt_cov64(d: int, exponent: float, seed: int, stream: int, bits: int = S_BITS) -> np.ndarray:
    """S = Q diag(lambda)^{1/2} (fp64), lambda_i = i^-exponent, so S S^T = Q diag(lambda) Q^T,
    on the 2^-bits grid (|S_ij| <= 1, since lambda_i <= 1 and Q is orthogonal)."""
    lam = np.arange(1, d + 1, dtype=np.float64) ** (-float(exponent))
    return _grid(orthogonal64(d, seed, stream) * np.sqrt(lam)[None, :], bits)


def _normals(seed: int, key: int, c: int, shape) -> np.ndarray:
    """Standard normal variates on the 2^-Z_BITS grid, clipped to |z| <= Z_CLIP."""
    return _grid(_rng(seed, key, c).standard_normal(shape), Z_BITS, Z_CLIP)


def _threads() -> int:
    try:
        n = len(os.sched_getaffinity(0))
    except Exception:
        n = os.cpu_count() or 1
    return max(1, min(16, n))


def _round_to(x64: torch.Tensor, dtype: torch.dtype) -> torch.Tensor:
    x32 = x64.to(torch.float32)
    return x32 if dtype == torch.float32 else x32.to(dtype)


def rank_one_samples(wl: Workload, seed: int = 0, device="cpu", N: Optional[int] = None):
    """(X, G) of the rank-one workload `wl` on `device`, dtype wl.dtype, drawn portably.

    x_k = S_x z_k (Gaussian) or S_x z_k / sqrt(w_k / nu) (multivariate Student-t,
    w_k a sum of nu squared normals), then the outlier channels are scaled;
    g_k = g_scale S_g z'_k.  The mixing is exact, the rest single IEEE fp64 operations,
    one rounding at the end."""
    assert wl.kind == "rank_one"
    N = wl.N if N is None else int(N)
    dev = torch.device(device)
    SxT = torch.from_numpy(sqrt_cov64(wl.n, wl.x_exponent, seed, _QX).T.copy()).to(dev)
    SgT = torch.from_numpy(sqrt_cov64(wl.m, wl.g_exponent, seed, _QG).T.copy()).to(dev)
    col = np.ones(wl.n)
    if wl.x_outliers:
        col[_rng(seed, _OUT).permutation(wl.n)[: wl.x_outliers]] = wl.outlier_scale
    col_t = torch.from_numpy(col).to(dev)
    X = torch.empty(N, wl.n, device=dev, dtype=wl.torch_dtype)
    G = torch.empty(N, wl.m, device=dev, dtype=wl.torch_dtype)
    nu = int(wl.student_nu)

    def draw(c: int):
        r0 = c * CHUNK_ROWS
        rows = min(N, r0 + CHUNK_ROWS) - r0
        zx = _normals(seed, _ZX, c, (rows, wl.n))
        zg = _normals(seed, _ZG, c, (rows, wl.m))
        f = None
        if nu:
            u = _rng(seed, _W, c).standard_normal((rows, nu))
            w = u[:, 0] * u[:, 0]
            for j in range(1, nu):          # fixed summation order
                w = w + u[:, j] * u[:, j]
            f = 1.0 / np.sqrt(w / nu)
        return r0, rows, zx, zg, f

    nchunks = (N + CHUNK_ROWS - 1) // CHUNK_ROWS
    with ThreadPoolExecutor(_threads()) as ex:
        ahead = max(2, _threads())
        futs = [ex.submit(draw, c) for c in range(min(nchunks, ahead))]
        for c in range(nchunks):
            r0, rows, zx, zg, f = futs[c].result()
            futs[c] = None
            if c + ahead < nchunks:
                futs.append(ex.submit(draw, c + ahead))
            x = torch.from_numpy(zx).to(dev) @ SxT
            if f is not None:
                x = x * torch.from_numpy(f).to(dev).unsqueeze(1)
            x = x * col_t
            X[r0:r0 + rows] = _round_to(x, wl.torch_dtype)
            g = (torch.from_numpy(zg).to(dev) @ SgT) * wl.g_scale
            G[r0:r0 + rows] = _round_to(g, wl.torch_dtype)
            del x, g
    return X, G


def matrix_normal_factors(wl: Workload, seed: int = 0):
    """(S_A, S_B) in fp64 on the host for the matrix workload: S S^T = A0 (n x n), B0
    (m x m), power-law spectra with condition number wl.cond (S_A on the coarser grid
    of the second, exact, product)."""
    SA = sqrt_cov64(wl.n, exponent_for_condition(wl.n, wl.cond), seed, _QA, bits=SA_BITS)
    SB = sqrt_cov64(wl.m, exponent_for_condition(wl.m, wl.cond), seed, _QB)
    return SA, SB


def matrix_sample_chunk(wl: Workload, seed: int, k0: int, k1: int, SA_t: torch.Tensor,
                        SB_t: torch.Tensor) -> torch.Tensor:
    """Samples k0..k1-1 of the matrix workload, G_k = S_B Z_k S_A^T (fp64 on the device
    of SA_t, rounded once to wl.dtype).  Y_k = S_B Z_k is exact and is put on the
    2^-Y_BITS grid (clipped to |y| <= Y_CLIP) before the second product, which is then
    exact too.  Samples are drawn per generator chunk of CHUNK_ROWS // 64 samples, so any
    k0..k1 reproduce the same bytes."""
    per = max(1, CHUNK_ROWS // 64)
    out = []
    dev = SA_t.device
    c0, c1 = k0 // per, (k1 - 1) // per
    for c in range(c0, c1 + 1):
        a = c * per
        rows = min(wl.N, a + per) - a
        z = _normals(seed, _ZK, c, (rows, wl.m, wl.n))
        lo, hi = max(k0, a) - a, min(k1, a + rows) - a
        zt = torch.from_numpy(z[lo:hi]).to(dev)
        y = torch.matmul(SB_t, zt).clamp_(-Y_CLIP, Y_CLIP)
        y = torch.round(y * (2.0 ** Y_BITS)) * (2.0 ** -Y_BITS)
        out.append(_round_to(torch.matmul(y, SA_t.t()), wl.torch_dtype))
    return torch.cat(out, 0)


def matrix_blocks(wl: Workload, seed: int = 0, device="cpu", N: Optional[int] = None):
    """Yield (k0, block) over all samples of the matrix workload in generator chunks of
    CHUNK_ROWS // 64 samples (G_k = S_B Z_k S_A^T exactly as matrix_sample_chunk), the
    normals of the next chunks drawn by a thread pool meanwhile."""
    assert wl.kind == "matrix"
    N = wl.N if N is None else int(N)
    dev = torch.device(device)
    SA, SB = matrix_normal_factors(wl, seed)
    SA_t, SB_t = torch.from_numpy(SA).to(dev), torch.from_numpy(SB).to(dev)
    per = max(1, CHUNK_ROWS // 64)
    nchunks = (N + per - 1) // per

    def draw(c):
        rows = min(N, (c + 1) * per) - c * per
        return _normals(seed, _ZK, c, (rows, wl.m, wl.n))

    with ThreadPoolExecutor(_threads()) as ex:
        ahead = max(2, _threads())
        futs = [ex.submit(draw, c) for c in range(min(nchunks, ahead))]
        for c in range(nchunks):
            z = futs[c].result()
            futs[c] = None
            if c + ahead < nchunks:
                futs.append(ex.submit(draw, c + ahead))
            y = torch.matmul(SB_t, torch.from_numpy(z).to(dev)).clamp_(-Y_CLIP, Y_CLIP)
            y = torch.round(y * (2.0 ** Y_BITS)) * (2.0 ** -Y_BITS)
            yield c * per, _round_to(torch.matmul(y, SA_t.t()), wl.torch_dtype)


def matrix_samples(wl: Workload, seed: int = 0, device="cpu", N: Optional[int] = None):
    """All N matrix samples (N x m x n, dtype wl.dtype) on `device`, drawn portably."""
    N = wl.N if N is None else int(N)
    out = torch.empty(N, wl.m, wl.n, dtype=wl.torch_dtype, device=device)
    for k0, blk in matrix_blocks(wl, seed, device, N):
        out[k0:k0 + blk.shape[0]] = blk
    return out


def sha256(*tensors: torch.Tensor, chunk_bytes: int = 1 << 28) -> str:
    """Digest of the raw bytes of the tensors, in order (row-major, as stored)."""
    h = hashlib.sha256()
    for t in tensors:
        flat = t.contiguous().view(-1).view(torch.uint8)
        for i in range(0, flat.numel(), chunk_bytes):
            h.update(flat[i:i + chunk_bytes].cpu().numpy().tobytes())
    return h.hexdigest()
