"""fp64 CPU oracle of the FlipFlop Hessian fit.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg, never by the library.  It shares no code with the CUDA path.
See flipflop.py (the fit) and waterkron.py (reverse Cholesky, waterfilling scales, two-sided
GPTQ) for what each function computes and the paper passages it follows.
"""
from .flipflop import (FitResult, as_f64, cholesky, damp, factor_rel_errs, flipflop_fit,
                       flipflop_fit_matrix, flipflop_fit_matrix_blocks, frobenius_fit, fwd_quad_forms, gaussian_loglik,
                       input_hessian, inv_quad_forms_chol, kron_rel_err, logdet_from_cholesky,
                       inv_quad_forms_rows, loglik, marginal_hessian, normalized, phi_tilde,
                       rel_change, row_blocks, tri_inverse, weighted_gram, weighted_gram_rows)
from . import waterkron

__all__ = ["FitResult", "as_f64", "cholesky", "damp", "factor_rel_errs", "flipflop_fit",
           "flipflop_fit_matrix", "flipflop_fit_matrix_blocks", "frobenius_fit", "fwd_quad_forms", "gaussian_loglik",
           "input_hessian", "inv_quad_forms_chol", "kron_rel_err", "logdet_from_cholesky",
           "inv_quad_forms_rows", "loglik", "marginal_hessian", "normalized", "phi_tilde",
           "rel_change", "row_blocks", "tri_inverse", "weighted_gram", "weighted_gram_rows",
           "waterkron"]
