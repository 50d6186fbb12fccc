"""Seeded synthetic inputs shared by the oracle's tests and the CUDA path's tests
and benchmark.  No estimator arithmetic lives here."""
from .workloads import (WORKLOADS, Workload, factorial_design, gaussian, matrix_normal_factors,
                        matrix_samples, rademacher, rank_one_samples, spd_matrix)

__all__ = ["WORKLOADS", "Workload", "factorial_design", "gaussian", "matrix_normal_factors",
           "matrix_samples", "rademacher", "rank_one_samples", "spd_matrix"]
