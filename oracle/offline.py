"""Oracle for the offline side of the method, in float64.

TEST INFRASTRUCTURE, like the rest of this package: imported only by the
tests; the product path never imports it.

  Sec. 4.1  "Chunk-cache preparation": each chunk is prefilled alone and its K
            is stored in canonical coordinates, K^c_t = R_M(q_t)^{-1} K_t with
            q_t the token's local position; V is stored as it is.
  Sec. 4.2  "Normalization and objective": sigma_stale and sigma_Delta are RMS
            values over corpus document tokens, separately for each target
            layer, KV head, K/V component and head coordinate, i.e. one value
            per D_KV coordinate.  sigma_stale is taken over stale caches,
            sigma_Delta over the residual targets KV_joint^c - KV_stale^c.

Reading (R17): the inverse rotation is the same
rotate-half rotation as R_M (R10) with the angle negated, computed exactly
and rounded once to the cache dtype (R11); the RMS is sqrt(mean of squares)
over all tokens given, without centring.
"""
from __future__ import annotations

from typing import Iterable, Optional

import numpy as np

from .cacherepair import dtype_to_f64, rope_rotate_half, round_to_cache

__all__ = ["canonical_exact", "canonicalize_chunk", "sigma_rms"]


def canonical_exact(kv: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray, *, n_layers: int,
                    n_kv_heads: int, head_dim: int, cache_dtype: str) -> np.ndarray:
    """K^c_t = R_M(q_t)^{-1} K_t on every K segment, V unchanged, exact (float64)."""
    n = kv.shape[0]
    x = dtype_to_f64(kv, cache_dtype).reshape(n, n_layers, 2, n_kv_heads, head_dim).copy()
    x[:, :, 0] = rope_rotate_half(x[:, :, 0], -np.asarray(pos, np.float64), inv_freq)
    return x.reshape(n, -1)


def canonicalize_chunk(kv: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray, *, n_layers: int,
                       n_kv_heads: int, head_dim: int, cache_dtype: str) -> np.ndarray:
    """The stored canonical cache: canonical_exact rounded once to the cache dtype."""
    return round_to_cache(canonical_exact(kv, pos, inv_freq, n_layers=n_layers,
                                          n_kv_heads=n_kv_heads, head_dim=head_dim,
                                          cache_dtype=cache_dtype), cache_dtype)


def sigma_rms(caches: Iterable[np.ndarray], cache_dtype: str,
              minus: Optional[Iterable[np.ndarray]] = None) -> np.ndarray:
    """Per-coordinate RMS over all tokens of `caches` (each [n_i, D_KV]); with
    `minus`, of the differences caches[i] - minus[i] (sigma_Delta)."""
    caches = list(caches)
    subs = list(minus) if minus is not None else [None] * len(caches)
    total, count = None, 0
    for a, b in zip(caches, subs):
        x = dtype_to_f64(a, cache_dtype)
        if b is not None:
            x = x - dtype_to_f64(b, cache_dtype)
        s = np.sum(x * x, axis=0)
        total = s if total is None else total + s
        count += x.shape[0]
    return np.sqrt(total / count)
