"""Seeded synthetic inputs shaped like the paper's workloads.

This module only draws random numbers (numpy PCG64 ``default_rng``); it holds
none of the method's arithmetic, so both the CUDA path and the CPU oracle may
use it.  The distributions stand in for the paper's synthetic vectors
(Normal, Lognormal, Student-t, sparse outliers) and for its real-model weight,
gradient and KV-cache tensors, which are not available here.
"""
from __future__ import annotations

import numpy as np


def normal(d: int, seed: int = 0) -> np.ndarray:
    """i.i.d. N(0, 1), fp32."""
    return np.random.default_rng(seed).standard_normal(d).astype(np.float32)


def signed_lognormal(d: int, seed: int = 0) -> np.ndarray:
    """sign * LogNormal(0, 1) with equiprobable signs (heavy-tailed, gradient-like)."""
    rng = np.random.default_rng(seed)
    mag = rng.lognormal(0.0, 1.0, d)
    sign = np.where(rng.random(d) < 0.5, -1.0, 1.0)
    return (sign * mag).astype(np.float32)


def student_t(d: int, seed: int = 0, df: float = 3.0, scale: float = 1e-3) -> np.ndarray:
    """scale * Student-t(df) (gradient-like)."""
    return (scale * np.random.default_rng(seed).standard_t(df, d)).astype(np.float32)


def kv_rows(rows: int, d: int, seed: int = 0, outlier_frac: float = 0.01) -> np.ndarray:
    """KV-cache-like rows: row r ~ N(0, sigma_r^2), sigma_r ~ U[0.1, 4]; each
    entry is independently replaced with probability outlier_frac by
    +-8 sigma_r (random sign).  Shape [rows, d], fp32."""
    rng = np.random.default_rng(seed)
    sig = rng.uniform(0.1, 4.0, rows)
    x = rng.standard_normal((rows, d)) * sig[:, None]
    hit = rng.random((rows, d)) < outlier_frac
    sgn = np.where(rng.random((rows, d)) < 0.5, -1.0, 1.0)
    x = np.where(hit, 8.0 * sgn * sig[:, None], x)
    return x.astype(np.float32)


def mixture(d: int, seed: int = 0) -> np.ndarray:
    """Weight-matrix-like mixture: w.p. 0.9 N(0, 1), else N(0, 10^2)."""
    rng = np.random.default_rng(seed)
    wide = rng.random(d) < 0.1
    x = rng.standard_normal(d) * np.where(wide, 10.0, 1.0)
    return x.astype(np.float32)


# The five workloads (single vectors unless noted): generator, d, s, budgets.
CONFIGS = {
    "normal_d1024_s8": dict(gen=normal, d=1024, s=8, budgets=(2.0,), refine=True),
    "lognormal_d16384_s16": dict(gen=signed_lognormal, d=16384, s=16, budgets=(1.0, 2.0, 3.0)),
    "studentt_d131072_s16": dict(gen=student_t, d=131072, s=16, budgets=(2.5,), refine=True,
                                 refine_tol=1e-9),
    "kvrows_8192x128_s8": dict(gen=kv_rows, rows=8192, d=128, s=8, budgets=(3.0,)),
    "mixture_d1048576_s32": dict(gen=mixture, d=1048576, s=32, budgets=(4.0,)),
}


def make(name: str, seed: int = 0) -> np.ndarray:
    c = CONFIGS[name]
    if "rows" in c:
        return c["gen"](c["rows"], c["d"], seed)
    return c["gen"](c["d"], seed)
