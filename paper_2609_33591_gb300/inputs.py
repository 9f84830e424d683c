"""Seeded synthetic inputs for K-interval attention.

This module only draws random numbers; it holds none of the operator's
arithmetic.  Both the CUDA path (tests, benchmark) and the CPU oracle read the
same fp32 arrays it returns.

Distributions follow the workloads the paper's attention layers see in shape
(GPT-2-small: 12 heads of d = 64 at T = 1024; a 1B-scale layer: d = 128) with
i.i.d. N(0, 1) entries for Q, K, V and dO.  The score scale 1/sqrt(d) of
Sec. 3 is applied inside the operator, not here.
"""
from __future__ import annotations

import numpy as np


def make_qkvdo(B: int, H: int, T: int, d: int, seed: int, *, peaked_frac: float = 0.0,
               peak_boost: float = 12.0) -> tuple[np.ndarray, np.ndarray, np.ndarray, np.ndarray]:
    """Q, K, V, dO as fp32 [B, H, T, d], drawn in that order from PCG64(seed).

    ``peaked_frac`` > 0 gives peaked rows: for each (b, h), floor(peaked_frac * T)
    distinct query rows i are chosen, each with one key j uniform in 0..i, and
    Q_i is moved along K_j so that the scaled score s_ij = Q_i . K_j / sqrt(d)
    rises by ``peak_boost`` (in exact arithmetic).
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    shape = (B, H, T, d)
    Q = rng.standard_normal(shape, dtype=np.float32)
    K = rng.standard_normal(shape, dtype=np.float32)
    V = rng.standard_normal(shape, dtype=np.float32)
    dO = rng.standard_normal(shape, dtype=np.float32)
    n_peak = int(np.floor(peaked_frac * T))
    if n_peak > 0:
        root_d = np.sqrt(np.float64(d))
        for b in range(B):
            for h in range(H):
                rows = rng.choice(T, size=n_peak, replace=False)
                for i in rows:
                    j = int(rng.integers(0, i + 1))
                    kj = K[b, h, j].astype(np.float64)
                    step = (peak_boost * root_d) * kj / float(kj @ kj)
                    Q[b, h, i] = (Q[b, h, i].astype(np.float64) + step).astype(np.float32)
    return Q, K, V, dO
