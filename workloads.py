"""Seeded synthetic inputs shared by the tests, the bench and the oracle runs.

This module holds the input recipe only -- none of the method's arithmetic.
The recipe follows the workloads the paper prices for dense DGEMM (§3, §4.1)
with the entry distribution a_ij = U(-1/2, 1/2) · exp(φ · N(0, 1)), i.i.d.,
drawn from numpy's PCG64 generator.  The paper measures on no public dataset
for this path; these seeded matrices stand in for its dense GEMM call shapes.

Matrices are returned in column-major (Fortran) order, as the C-ABI expects.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np


@dataclass(frozen=True)
class Workload:
    name: str
    m: int
    n: int
    k: int
    phi: float
    r: int
    scaled_rows: float = 0.0     # fraction of A's rows scaled by 2^±300
    index: int = 0               # seeds: A = 1000 + index, B = 2000 + index

    @property
    def flops(self) -> float:
        return 2.0 * self.m * self.n * self.k


# The five dense shapes: a small case the oracle finishes in seconds, the
# square 4096 case, the square 16384 ceiling case, a tall-K case stressing
# K-chunking, and a k = 64 case with a wide dynamic range and 1% of A's rows
# scaled by 2^±300 (native-FP64 fallback rows); a batched-GEMV shape; and a
# small-C, long-k shape.
WORKLOADS = {
    "dgemm_256": Workload("dgemm_256", 256, 256, 256, 0.5, 12, index=1),
    "dgemm_4096": Workload("dgemm_4096", 4096, 4096, 4096, 0.5, 12, index=2),
    "dgemm_16384": Workload("dgemm_16384", 16384, 16384, 16384, 1.0, 13, index=3),
    "dgemm_tallk": Workload("dgemm_tallk", 1024, 1024, 65536, 0.5, 12, index=4),
    "dgemm_k64_wide": Workload("dgemm_k64_wide", 16384, 16384, 64, 4.0, 12,
                               scaled_rows=0.01, index=5),
    # Batched GEMV (§3 "Strategy 1"): Y = A·X with a batch of 16 right-hand
    # sides, through the same kernels.
    "gemv_batch16": Workload("gemv_batch16", 16384, 16, 16384, 0.5, 12, index=6),
    # A Gram-type block: a small C with a long k, which the residue GEMM
    # splits along k.
    "gram_256": Workload("gram_256", 256, 256, 65536, 0.5, 12, index=7),
}


def random_matrix(rows: int, cols: int, phi: float, seed: int) -> np.ndarray:
    """rows × cols float64, a = U(-1/2, 1/2)·exp(φ N(0,1)), column-major."""
    rng = np.random.default_rng(seed)
    u = rng.uniform(-0.5, 0.5, size=(cols, rows))
    g = rng.standard_normal(size=(cols, rows))
    x = u * np.exp(phi * g)
    return x.T  # transpose of a C-ordered (cols, rows) array is Fortran-ordered


def scale_rows(A: np.ndarray, fraction: float, seed: int) -> np.ndarray:
    """Scale a seeded choice of ⌈fraction·m⌉ rows: half by 2^300, half by 2^-300."""
    m = A.shape[0]
    cnt = int(np.ceil(fraction * m)) if fraction > 0 else 0
    if cnt == 0:
        return A
    rng = np.random.default_rng(seed)
    rows = np.sort(rng.choice(m, size=cnt, replace=False))
    A = np.asfortranarray(A.copy())
    A[rows[: cnt // 2], :] *= 2.0 ** 300
    A[rows[cnt // 2:], :] *= 2.0 ** -300
    return A


def make_inputs(w: Workload, m: int = None, n: int = None, k: int = None):
    """(A, B) for a workload; sizes may be overridden for reduced test cases."""
    m = w.m if m is None else m
    n = w.n if n is None else n
    k = w.k if k is None else k
    A = random_matrix(m, k, w.phi, 1000 + w.index)
    B = random_matrix(k, n, w.phi, 2000 + w.index)
    if w.scaled_rows:
        A = scale_rows(A, w.scaled_rows, 3000 + w.index)
    return A, B
