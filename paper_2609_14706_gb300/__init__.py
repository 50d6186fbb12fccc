"""FlipFlop Hessian estimator on one GB300 GPU: Python binding of libffh.

This module only marshals arguments to the C ABI declared in include/ffh.h; every
step of the fit runs in the library's CUDA kernels.  There is no CPU fallback: if
libffh.so is missing or no sm_100-family GPU is present, calls raise.

    import paper_2609_14706_gb300 as ffh
    with ffh.Handle(dtype="bf16") as h:
        A, B = h.fit(X, G, iters=8)          # X: N x n, G: N x m (torch tensors)
        stats = h.stats()
"""
from __future__ import annotations

import ctypes
import math
import os
import re
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libffh.so")
HEADER_PATH = os.path.join(os.path.dirname(_HERE), "include", "ffh.h")

STATUS = {0: "FFH_OK", 1: "FFH_ERR_INVALID_ARG", 2: "FFH_ERR_NOT_SPD", 3: "FFH_ERR_RANK",
          4: "FFH_ERR_OOM", 5: "FFH_ERR_CUDA", 6: "FFH_ERR_TIMEOUT", 7: "FFH_ERR_UNSUPPORTED"}
FFH_BF16, FFH_F32 = 0, 1
FFH_FLIPFLOP, FFH_FROBENIUS, FFH_INPUT, FFH_MARGINAL = 0, 1, 2, 3
VARIANTS = {"flipflop": FFH_FLIPFLOP, "frobenius": FFH_FROBENIUS, "input": FFH_INPUT,
            "marginal": FFH_MARGINAL}
FAULT_NONE, FAULT_OOM, FAULT_BAD_PIVOT, FAULT_LOST_COPY = 0, 1, 2, 3


class ffh_options(ctypes.Structure):
    _fields_ = [("dtype", ctypes.c_int32), ("damping", ctypes.c_float),
                ("variant", ctypes.c_int32), ("init_A", ctypes.c_void_p),
                ("final_loglik", ctypes.c_int32), ("reserved0", ctypes.c_int32),
                ("fault", ctypes.c_int32), ("profile", ctypes.c_int32),
                ("no_graph", ctypes.c_int32), ("reserved", ctypes.c_int32 * 3)]


class ffh_timings(ctypes.Structure):
    _fields_ = [("gram_ms", ctypes.c_double), ("gram_launches", ctypes.c_int64),
                ("qform_ms", ctypes.c_double), ("qform_launches", ctypes.c_int64),
                ("chol_ms", ctypes.c_double), ("chol_calls", ctypes.c_int64),
                ("kernel_launches", ctypes.c_int64)]


class FFHError(RuntimeError):
    def __init__(self, code: int, where: str, msg: str):
        self.code = code
        self.status = STATUS.get(code, str(code))
        super().__init__(f"{where}: {self.status}: {msg}")


_lib = None


def load_library(path: Optional[str] = None):
    """Load libffh.so (built in-tree by build.build()).  Raises if it is missing."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(f"{p} is not built; run paper_2609_14706_gb300.build.build() "
                           "(or __graft_entry__.build())")
    lib = ctypes.CDLL(p)
    vp, i64, i32, f32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float
    pd, pi = ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_int32)
    sigs = {
        "ffh_version": ([], i32),
        "ffh_create": ([ctypes.POINTER(vp), ctypes.POINTER(ffh_options), vp], ctypes.c_int),
        "ffh_set_options": ([vp, ctypes.POINTER(ffh_options)], ctypes.c_int),
        "ffh_set_stream": ([vp, vp], ctypes.c_int),
        "ffh_destroy": ([vp], ctypes.c_int),
        "ffh_last_error": ([vp], ctypes.c_char_p),
        "ffh_fit": ([vp, vp, vp, i64, i64, i64, i32, f32, vp, vp], ctypes.c_int),
        "ffh_fit_matrix": ([vp, vp, i64, i64, i64, i32, f32, vp, vp], ctypes.c_int),
        "ffh_get_stats": ([vp, pi, pd, pd, pd, i32, pi], ctypes.c_int),
        "ffh_weighted_gram": ([vp, vp, vp, i64, i64, f32, vp], ctypes.c_int),
        "ffh_quad_form": ([vp, vp, vp, i64, i64, vp], ctypes.c_int),
        "ffh_cholesky": ([vp, vp, i64, vp, vp, pd], ctypes.c_int),
        "ffh_get_timings": ([vp, ctypes.POINTER(ffh_timings), i32], ctypes.c_int),
        "ffh_weighted_gram_static": ([vp, vp, i64, i64, f32, vp, vp, ctypes.c_char_p, i32],
                                     ctypes.c_int),
        "ffh_phi_tilde": ([vp, vp, vp, i64, i64, i64, vp, vp, pd], ctypes.c_int),
        "ffh_rev_cholesky": ([vp, vp, i64, vp, vp, pd], ctypes.c_int),
        "ffh_waterfilling_scales": ([vp, vp, i64, vp, i64, f32, vp, vp], ctypes.c_int),
        "ffh_gptq2": ([vp, vp, vp, vp, vp, vp, i64, i64, vp, vp], ctypes.c_int),
        "ffh_partial_gram": ([vp, vp, vp, i64, i64, i64, vp, i32, vp, pd], ctypes.c_int),
        "ffh_update_from_sum": ([vp, vp, i64, ctypes.c_double, vp], ctypes.c_int),
        "ffh_normalize_pair": ([vp, vp, i64, vp, i64, pd], ctypes.c_int),
        "ffh_relative_change": ([vp, vp, vp, i64, pd], ctypes.c_int),
    }
    for name, (args, res) in sigs.items():
        fn = getattr(lib, name)
        fn.argtypes = args
        fn.restype = res
    if path is None:
        _lib = lib
    return lib


def header_symbols(path: str = HEADER_PATH):
    """Names of the functions declared in include/ffh.h."""
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ffh_[a-z_]+)\s*\(", text)))


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _check(lib, h, code: int, where: str):
    if code != 0:
        msg = lib.ffh_last_error(h).decode() if h else ""
        raise FFHError(code, where, msg)


def _dtype_code(dtype) -> int:
    if dtype in ("bf16", torch.bfloat16, FFH_BF16):
        return FFH_BF16
    if dtype in ("f32", "fp32", torch.float32, FFH_F32):
        return FFH_F32
    raise ValueError(f"unsupported dtype {dtype}")


class Handle:
    """One libffh handle: options, a CUDA stream and a device workspace."""

    def __init__(self, dtype="bf16", damping: float = 0.0, variant: str = "flipflop",
                 init_A: Optional[torch.Tensor] = None, final_loglik: bool = False,
                 fault: int = 0, profile: bool = False,
                 stream: Optional[torch.cuda.Stream] = None, graph: bool = True):
        self._lib = load_library()
        self._keep = []
        self.opts = ffh_options()
        self.opts.dtype = _dtype_code(dtype)
        self.opts.damping = float(damping)
        self.opts.variant = VARIANTS[variant]
        if init_A is not None:
            init_A = init_A.to(torch.float32).contiguous()
            self._keep.append(init_A)
            self.opts.init_A = init_A.data_ptr()
        self.opts.final_loglik = int(bool(final_loglik))
        self.opts.fault = int(fault)
        self.opts.profile = int(bool(profile))
        self.opts.no_graph = 0 if graph else 1
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        self._h = ctypes.c_void_p()
        code = self._lib.ffh_create(ctypes.byref(self._h), ctypes.byref(self.opts),
                                    ctypes.c_void_p(self.stream.cuda_stream))
        _check(self._lib, None, code, "ffh_create")

    # -- lifetime --
    def close(self):
        if self._h:
            self._lib.ffh_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _sample_dtype(self):
        return torch.bfloat16 if self.opts.dtype == FFH_BF16 else torch.float32

    def _samples(self, V: torch.Tensor, name: str) -> torch.Tensor:
        if V.dtype != self._sample_dtype():
            raise TypeError(f"{name} must be {self._sample_dtype()} for this handle, got {V.dtype}")
        return V.contiguous()

    # -- the fit --
    def fit(self, X: torch.Tensor, G: torch.Tensor, iters: int, tol: float = 0.0,
            A_out: Optional[torch.Tensor] = None, B_out: Optional[torch.Tensor] = None):
        """ffh_fit: A (n x n, tr A = n) and B (m x m) fitted to rows x_k of X, g_k of G."""
        X, G = self._samples(X, "X"), self._samples(G, "G")
        N, n = X.shape
        m = G.shape[1]
        dev = X.device
        if A_out is None:
            A_out = torch.empty(n, n, dtype=torch.float32, device=dev)
        if B_out is None:
            B_out = torch.empty(m, m, dtype=torch.float32, device=dev)
        code = self._lib.ffh_fit(self._h, _ptr(X), _ptr(G), N, n, m, int(iters), float(tol),
                                 _ptr(A_out), _ptr(B_out))
        _check(self._lib, self._h, code, "ffh_fit")
        return A_out, B_out

    def fit_matrix(self, Gk: torch.Tensor, iters: int, tol: float = 0.0,
                   A_out: Optional[torch.Tensor] = None, B_out: Optional[torch.Tensor] = None):
        """ffh_fit_matrix: fit to matrix samples Gk (N x m x n, fp32)."""
        if Gk.dtype != torch.float32:
            raise TypeError("Gk must be float32")
        Gk = Gk.contiguous()
        N, m, n = Gk.shape
        dev = Gk.device
        if A_out is None:
            A_out = torch.empty(n, n, dtype=torch.float32, device=dev)
        if B_out is None:
            B_out = torch.empty(m, m, dtype=torch.float32, device=dev)
        code = self._lib.ffh_fit_matrix(self._h, _ptr(Gk), N, n, m, int(iters), float(tol),
                                        _ptr(A_out), _ptr(B_out))
        _check(self._lib, self._h, code, "ffh_fit_matrix")
        return A_out, B_out

    def stats(self, capacity: int = 4096) -> dict:
        """ffh_get_stats of the last fit."""
        it = ctypes.c_int32()
        delta = ctypes.c_double()
        ntr = ctypes.c_int32()
        ll = (ctypes.c_double * capacity)()
        mqr = (ctypes.c_double * capacity)()
        code = self._lib.ffh_get_stats(self._h, ctypes.byref(it), ctypes.byref(delta), ll, mqr,
                                       capacity, ctypes.byref(ntr))
        _check(self._lib, self._h, code, "ffh_get_stats")
        k = min(ntr.value, capacity)
        return {"iters_done": it.value, "delta": delta.value, "loglik": list(ll[:k]),
                "mean_qr": list(mqr[:k])}

    def timings(self, reset: bool = False) -> dict:
        """ffh_get_timings: kernel times accumulated while profile=True."""
        t = ffh_timings()
        code = self._lib.ffh_get_timings(self._h, ctypes.byref(t), int(bool(reset)))
        _check(self._lib, self._h, code, "ffh_get_timings")
        return {f: getattr(t, f) for f, _ in ffh_timings._fields_}

    def phi_tilde(self, X: torch.Tensor, G: torch.Tensor, A: torch.Tensor,
                  B: torch.Tensor) -> float:
        """ffh_phi_tilde: scale-free mismatch factor of A (x) B on the samples."""
        X, G = self._samples(X, "X"), self._samples(G, "G")
        N, n = X.shape
        m = G.shape[1]
        A = A.to(torch.float32).contiguous()
        B = B.to(torch.float32).contiguous()
        out = ctypes.c_double()
        code = self._lib.ffh_phi_tilde(self._h, _ptr(X), _ptr(G), N, n, m, _ptr(A), _ptr(B),
                                       ctypes.byref(out))
        _check(self._lib, self._h, code, "ffh_phi_tilde")
        return out.value

    # -- single steps --
    def weighted_gram(self, V: torch.Tensor, w: Optional[torch.Tensor], scale: float = 1.0,
                      C_out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """ffh_weighted_gram: scale * V^T diag(w) V (w None: unweighted)."""
        V = self._samples(V, "V")
        N, d = V.shape
        if w is not None:
            w = w.to(torch.float32).contiguous()
        if C_out is None:
            C_out = torch.empty(d, d, dtype=torch.float32, device=V.device)
        code = self._lib.ffh_weighted_gram(self._h, _ptr(V), _ptr(w), N, d, float(scale),
                                           _ptr(C_out))
        _check(self._lib, self._h, code, "ffh_weighted_gram")
        return C_out

    def quad_form(self, V: torch.Tensor, Linv: torch.Tensor,
                  q_out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """ffh_quad_form: q_k = ||Linv v_k||^2."""
        V = self._samples(V, "V")
        N, d = V.shape
        Linv = Linv.to(torch.float32).contiguous()
        if q_out is None:
            q_out = torch.empty(N, dtype=torch.float32, device=V.device)
        code = self._lib.ffh_quad_form(self._h, _ptr(V), _ptr(Linv), N, d, _ptr(q_out))
        _check(self._lib, self._h, code, "ffh_quad_form")
        return q_out

    def cholesky(self, F: torch.Tensor, want_inverse: bool = True):
        """ffh_cholesky: (L, L^-1 or None, log|F|)."""
        F = F.to(torch.float32).contiguous()
        d = F.shape[0]
        L = torch.empty_like(F)
        Li = torch.empty_like(F) if want_inverse else None
        ld = ctypes.c_double()
        code = self._lib.ffh_cholesky(self._h, _ptr(F), d, _ptr(L), _ptr(Li), ctypes.byref(ld))
        _check(self._lib, self._h, code, "ffh_cholesky")
        return L, Li, ld.value

    # ---- sample-sharded fit steps ----
    def partial_gram(self, U: torch.Tensor, V: torch.Tensor, F: Optional[torch.Tensor],
                     P_out: Optional[torch.Tensor] = None, accumulate: bool = False):
        """ffh_partial_gram: (P = sum_k (u_k^T F^-1 u_k) v_k v_k^T over these rows, log|F|);
        F None means F = I; accumulate adds P into P_out."""
        U, V = self._samples(U, "U"), self._samples(V, "V")
        N, du = U.shape
        dv = V.shape[1]
        if F is not None:
            F = F.to(torch.float32).contiguous()
        if P_out is None:
            if accumulate:
                raise ValueError("accumulate needs P_out")
            P_out = torch.empty(dv, dv, dtype=torch.float32, device=V.device)
        ld = ctypes.c_double()
        code = self._lib.ffh_partial_gram(self._h, _ptr(U), _ptr(V), N, du, dv, _ptr(F),
                                          int(bool(accumulate)), _ptr(P_out), ctypes.byref(ld))
        _check(self._lib, self._h, code, "ffh_partial_gram")
        return P_out, ld.value

    def update_from_sum(self, P: torch.Tensor, scale: float,
                        F_out: Optional[torch.Tensor] = None) -> torch.Tensor:
        """ffh_update_from_sum: damp(scale * P) with the handle's damping."""
        P = P.contiguous()
        if F_out is None:
            F_out = torch.empty_like(P)
        code = self._lib.ffh_update_from_sum(self._h, _ptr(P), P.shape[0], float(scale),
                                             _ptr(F_out))
        _check(self._lib, self._h, code, "ffh_update_from_sum")
        return F_out

    def normalize_pair(self, A: torch.Tensor, B: torch.Tensor) -> float:
        """ffh_normalize_pair: A /= s, B *= s with s = tr(A)/n (in place); returns s."""
        out = ctypes.c_double()
        code = self._lib.ffh_normalize_pair(self._h, _ptr(A), A.shape[0], _ptr(B), B.shape[0],
                                            ctypes.byref(out))
        _check(self._lib, self._h, code, "ffh_normalize_pair")
        return out.value

    def relative_change(self, F: torch.Tensor, Fprev: torch.Tensor) -> float:
        """ffh_relative_change: ||F/trF - P/trP||_F / ||F/trF||_F."""
        out = ctypes.c_double()
        code = self._lib.ffh_relative_change(self._h, _ptr(F), _ptr(Fprev), F.shape[0],
                                             ctypes.byref(out))
        _check(self._lib, self._h, code, "ffh_relative_change")
        return out.value

    # ---- WaterKron downstream (Sections 2-3) ----
    def rev_cholesky(self, F: torch.Tensor):
        """ffh_rev_cholesky: (L with L^T L = F, column-normalised L^-1, log|F|)."""
        F = F.to(torch.float32).contiguous()
        d = F.shape[0]
        L = torch.empty_like(F)
        Lt = torch.empty_like(F)
        ld = ctypes.c_double()
        code = self._lib.ffh_rev_cholesky(self._h, _ptr(F), d, _ptr(L), _ptr(Lt), ctypes.byref(ld))
        _check(self._lib, self._h, code, "ffh_rev_cholesky")
        return L, Lt, ld.value

    def waterfilling_scales(self, LA: torch.Tensor, LB: torch.Tensor, gamma: float):
        """ffh_waterfilling_scales: (alpha, beta) of Corollary 3.2."""
        LA, LB = LA.to(torch.float32).contiguous(), LB.to(torch.float32).contiguous()
        n, m = LA.shape[0], LB.shape[0]
        alpha = torch.empty(n, dtype=torch.float32, device=LA.device)
        beta = torch.empty(m, dtype=torch.float32, device=LA.device)
        code = self._lib.ffh_waterfilling_scales(self._h, _ptr(LA), n, _ptr(LB), m, float(gamma),
                                                 _ptr(alpha), _ptr(beta))
        _check(self._lib, self._h, code, "ffh_waterfilling_scales")
        return alpha, beta

    def gptq2(self, W: torch.Tensor, LtA: torch.Tensor, LtB: torch.Tensor, alpha: torch.Tensor,
              beta: torch.Tensor, want_v: bool = True):
        """ffh_gptq2 (Algorithm 2): (Z int32, V = beta alpha^T (.) Z or None)."""
        W = W.to(torch.float32).contiguous()
        m, n = W.shape
        Z = torch.empty(m, n, dtype=torch.int32, device=W.device)
        V = torch.empty(m, n, dtype=torch.float32, device=W.device) if want_v else None
        args = [t.to(torch.float32).contiguous() for t in (LtA, LtB, alpha, beta)]
        code = self._lib.ffh_gptq2(self._h, _ptr(W), *[_ptr(t) for t in args], m, n, _ptr(Z),
                                   _ptr(V))
        _check(self._lib, self._h, code, "ffh_gptq2")
        return Z, V


def waterkron_quantize(W: torch.Tensor, A: torch.Tensor, B: torch.Tensor, gamma: float,
                       handle: Optional["Handle"] = None):
    """Two-sided GPTQ of W (m x n) under A (x) B with the waterfilling scales:
    RevCholesky(A), RevCholesky(B) -> (alpha, beta) (Corollary 3.2) -> Algorithm 2.
    Returns (Z, V, alpha, beta)."""
    own = handle is None
    h = handle or Handle()
    try:
        LA, LtA, _ = h.rev_cholesky(A)
        LB, LtB, _ = h.rev_cholesky(B)
        alpha, beta = h.waterfilling_scales(LA, LB, gamma)
        Z, V = h.gptq2(W, LtA, LtB, alpha, beta)
        return Z, V, alpha, beta
    finally:
        if own:
            h.close()


def weighted_gram_static(V: torch.Tensor, w: Optional[torch.Tensor], scale: float = 1.0,
                         C_out: Optional[torch.Tensor] = None,
                         stream: Optional[torch.cuda.Stream] = None) -> torch.Tensor:
    """ffh_weighted_gram_static: scale * V^T diag(w) V with no device allocation by the
    library (bf16 V on the device; see include/ffh.h for the limits)."""
    lib = load_library()
    if V.dtype != torch.bfloat16:
        raise TypeError("V must be bfloat16")
    V = V.contiguous()
    N, d = V.shape
    if w is not None:
        w = w.to(torch.float32).contiguous()
    if C_out is None:
        C_out = torch.empty(d, d, dtype=torch.float32, device=V.device)
    stream = stream if stream is not None else torch.cuda.current_stream()
    buf = ctypes.create_string_buffer(256)
    code = lib.ffh_weighted_gram_static(_ptr(V), _ptr(w), N, d, float(scale), _ptr(C_out),
                                        ctypes.c_void_p(stream.cuda_stream), buf, 256)
    if code != 0:
        raise FFHError(code, "ffh_weighted_gram_static", buf.value.decode())
    return C_out


def fit(X: torch.Tensor, G: torch.Tensor, iters: int, tol: float = 0.0, **options):
    """One-shot ffh_fit with a temporary handle; returns (A, B, stats)."""
    dtype = "bf16" if X.dtype == torch.bfloat16 else "f32"
    with Handle(dtype=dtype, **options) as h:
        A, B = h.fit(X, G, iters, tol)
        return A, B, h.stats()


def fit_matrix(Gk: torch.Tensor, iters: int, tol: float = 0.0, **options):
    with Handle(dtype="f32", **options) as h:
        A, B = h.fit_matrix(Gk, iters, tol)
        return A, B, h.stats()


def gram_flops(N: int, d: int) -> float:
    """Algorithmic flops of one weighted Gram (lower triangle incl. diagonal)."""
    return float(N) * d * (d + 1)


def qform_flops(N: int, d: int) -> float:
    """Algorithmic flops of one triangular quadratic-form pass (N d (d+1))."""
    return float(N) * d * (d + 1)


def iteration_flops(N: int, n: int, m: int) -> float:
    """Algorithmic flops of one flip-flop iteration (two Grams, two quadratic forms)."""
    return gram_flops(N, n) + gram_flops(N, m) + qform_flops(N, n) + qform_flops(N, m)


__all__ = ["Handle", "FFHError", "fit", "fit_matrix", "weighted_gram_static", "load_library", "header_symbols",
           "gram_flops", "qform_flops", "iteration_flops", "ffh_options"]
