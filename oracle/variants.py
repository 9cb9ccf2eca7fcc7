"""Oracle for the output choices of the repair forward, in float64.

TEST INFRASTRUCTURE, like the rest of this package: imported only by the
tests; the product path never imports it.

  Sec. 2.2  The stale cache: the selected chunk caches, aligned to their
            request positions by re-rotating K, then concatenated.  With
            canonical chunk caches (Sec. 4.1) the re-rotation is R_M(p_t) on
            every K segment; this is also the "Stale KV" row of the
            experiments.
  App. F    Output choices ("Applying the predicted K and V"): the predicted
            correction applied to K only or to V only, the other component
            keeping its stale value; the first chunk keeping its stale cache;
            and ablation A5, where the head predicts the joint cache itself
            (zero output offset), whose normalised target is
            KV^c_joint / sigma_Delta.

Readings:
  R19 Under an output choice, every coordinate that is not repaired keeps its
      stale value exactly; with the target's R_M every K segment still leaves
      rotated, repaired or not (the other component's "stale value" is that of
      the stale cache above, whose K is rotated).
  R20 A5 (zero offset): the repaired value is sigma_Delta * z, formed exactly
      and rounded once to the cache dtype (R11), in place of
      KV_stale + sigma_Delta * z.
"""
from __future__ import annotations

from typing import Optional

import numpy as np

from .cacherepair import dtype_to_f64, global_rope_k, round_to_cache

__all__ = ["COMPONENTS", "OFFSETS", "component_columns", "apply_output_choice",
           "stale_kv_cache_exact", "stale_kv_cache"]

COMPONENTS = ("kv", "k", "v")
OFFSETS = ("stale", "zero")


def component_columns(component: str, *, n_layers: int, n_kv_heads: int, head_dim: int) -> np.ndarray:
    """Boolean [D_KV]: the coordinates of K (kv index 0), of V (1), or of both (R9)."""
    j = np.arange(n_layers * 2 * n_kv_heads * head_dim)
    kind = (j // (n_kv_heads * head_dim)) % 2         # j = ((l*2 + kind)*H + h)*d_h + d
    if component == "kv":
        return np.ones_like(j, bool)
    if component == "k":
        return kind == 0
    if component == "v":
        return kind == 1
    raise ValueError(f"unknown component {component!r}")


def apply_output_choice(kv: np.ndarray, z: np.ndarray, sigma_delta: np.ndarray, *, cache_dtype: str,
                        n_layers: int, n_kv_heads: int, head_dim: int, component: str = "kv",
                        offset: str = "stale", keep_rows: Optional[np.ndarray] = None,
                        pos: Optional[np.ndarray] = None,
                        inv_freq_target: Optional[np.ndarray] = None) -> np.ndarray:
    """The exact (float64) output cache of one request under an output choice.

    kv: the assembled stale cache (canonical K) in its stored dtype, [N, D_KV];
    z: the head output, [N, D_KV] float64; keep_rows: boolean [N], rows that keep
    their stale cache (the first chunk's rows for "keep first chunk").  With
    inv_freq_target every K segment is rotated by R_M(pos) at the end (R10, R19).
    """
    if offset not in OFFSETS:
        raise ValueError(f"unknown offset {offset!r}")
    stale = dtype_to_f64(kv, cache_dtype)
    corr = np.asarray(sigma_delta, np.float64)[None, :] * z
    repaired = stale + corr if offset == "stale" else corr
    sel = component_columns(component, n_layers=n_layers, n_kv_heads=n_kv_heads, head_dim=head_dim)
    out = np.where(sel[None, :], repaired, stale)
    if keep_rows is not None:
        out = np.where(np.asarray(keep_rows, bool)[:, None], stale, out)
    if inv_freq_target is not None:
        out = global_rope_k(out, pos, inv_freq_target, n_layers, n_kv_heads, head_dim)
    return out


def stale_kv_cache_exact(kv: np.ndarray, pos: np.ndarray, inv_freq_target: np.ndarray, *,
                         cache_dtype: str, n_layers: int, n_kv_heads: int, head_dim: int) -> np.ndarray:
    """The stale cache of Sec. 2.2 from canonical chunk caches: R_M(p_t) on K, exact."""
    return global_rope_k(dtype_to_f64(kv, cache_dtype), pos, inv_freq_target, n_layers,
                         n_kv_heads, head_dim)


def stale_kv_cache(kv: np.ndarray, pos: np.ndarray, inv_freq_target: np.ndarray, *, cache_dtype: str,
                   n_layers: int, n_kv_heads: int, head_dim: int) -> np.ndarray:
    """stale_kv_cache_exact rounded once to the cache dtype (R11)."""
    return round_to_cache(stale_kv_cache_exact(kv, pos, inv_freq_target, cache_dtype=cache_dtype,
                                               n_layers=n_layers, n_kv_heads=n_kv_heads,
                                               head_dim=head_dim), cache_dtype)
