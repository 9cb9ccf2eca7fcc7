"""Helpers for the GPU parity tests: device transfer and the tolerance checks.

Tolerances (written here once, used by every GPU test):
  * repaired K/V (the path's output): for every (layer, K|V) group,
        max_i  max(0, |gpu_i - exact_i| - ulp_cache(exact_i) / 2)  <=  2e-2 * RMS(exact)
    and cosine(gpu, exact) >= 0.999, where `exact` is the oracle's float64
    repaired value before rounding.  The half-ulp term admits the final
    rounding to the cache dtype, which both sides must do and which is coarser
    than the tolerance for large bf16 values (one bf16 ulp is 2^-7 relative).
  * integer and byte outputs (assembly, chunk map): bit-exact.
  * intermediate activations (diagnostics of each step): relative RMS error
    and max error relative to the reference RMS, thresholds per step below.
"""
import numpy as np
import torch

import oracle as O


def to_dev(a: np.ndarray, device="cuda") -> torch.Tensor:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(a).to(device)


def to_host(t: torch.Tensor) -> np.ndarray:
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def as_f64(a: np.ndarray) -> np.ndarray:
    if a.dtype == np.uint16:
        return O.dtype_to_f64(a, "bf16")
    return a.astype(np.float64)


def rel_errors(got: np.ndarray, want: np.ndarray):
    got, want = as_f64(got), as_f64(want)
    rms = np.sqrt(np.mean(want ** 2)) + 1e-300
    d = got - want
    return float(np.sqrt(np.mean(d ** 2)) / rms), float(np.abs(d).max() / rms)


def assert_close(got, want, rel_rms: float, max_rel: float, what=""):
    r, m = rel_errors(got, want)
    assert r <= rel_rms and m <= max_rel, f"{what}: rel-RMS {r:.3e} (<= {rel_rms}), max/RMS {m:.3e} (<= {max_rel})"
    return r, m


def assert_close_bf16(got, want, rel_rms: float = 3e-3, what=""):
    """A bf16 output: elementwise |err| <= 2^-8 |want| + 2e-3 RMS(want) (one rounding
    of the output plus fp32 accumulation order), and relative RMS error <= rel_rms."""
    g, w = as_f64(got), as_f64(want)
    rms = np.sqrt(np.mean(w ** 2))
    bad = np.abs(g - w) > np.abs(w) * 2.0 ** -8 + 2e-3 * rms
    r, m = rel_errors(got, want)
    assert not bad.any() and r <= rel_rms, f"{what}: {int(bad.sum())} elements out of bound, rel-RMS {r:.3e}, max/RMS {m:.3e}"
    return r, m


def half_ulp(x: np.ndarray, cache_dtype: str) -> np.ndarray:
    """Half a unit in the last place of x in the cache dtype (normal range)."""
    a = np.abs(x)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    mant = 7 if cache_dtype == "bf16" else 23
    return np.where(a > 0, np.exp2(e - mant - 1), 0.0)


def check_repaired_cache(got: np.ndarray, exact: np.ndarray, target, cache_dtype: str,
                         max_tol=2e-2, cos_tol=0.999, stale=None, resid_cos_tol=0.999):
    """The repaired-cache tolerance per (layer, K|V) group.

    Every group is measured before any assertion, so a failure reports the whole
    table.  With `stale` given (the un-repaired cache, canonical K), the residual
    alone (repaired - stale) is compared as well: its cosine per group must reach
    resid_cos_tol, which catches a wrong but small correction that the cache
    tolerance cannot see.  Returns (worst max err / RMS, worst cosine, worst
    residual cosine or None, rows), rows = (layer, 'K'|'V', err, cos, resid_cos).
    """
    g = as_f64(got) if cache_dtype == "bf16" else got.astype(np.float64)
    n = g.shape[0]
    L, H, dh = target.n_layers, target.n_kv_heads, target.head_dim
    g5 = g.reshape(n, L, 2, H * dh)
    e5 = exact.reshape(n, L, 2, H * dh)
    hu5 = half_ulp(exact, cache_dtype).reshape(n, L, 2, H * dh)
    s5 = None
    if stale is not None:
        s5 = (as_f64(stale) if cache_dtype == "bf16" else stale.astype(np.float64)).reshape(n, L, 2, H * dh)
    rows = []
    for l in range(L):
        for kv in range(2):
            gg, ee, hu = g5[:, l, kv], e5[:, l, kv], hu5[:, l, kv]
            rms = np.sqrt(np.mean(ee ** 2))
            err = float(np.maximum(np.abs(gg - ee) - hu, 0.0).max() / rms)
            cos = float((gg * ee).sum() / np.sqrt((gg ** 2).sum() * (ee ** 2).sum()))
            rc = None
            if s5 is not None:
                dg, de = gg - s5[:, l, kv], ee - s5[:, l, kv]
                rc = float((dg * de).sum() / np.sqrt((dg ** 2).sum() * (de ** 2).sum()))
            rows.append((l, "KV"[kv], err, cos, rc))
    worst_max = max(r[2] for r in rows)
    worst_cos = min(r[3] for r in rows)
    worst_rc = min(r[4] for r in rows) if s5 is not None else None
    for l, kv, err, cos, rc in rows:
        assert err <= max_tol, f"layer {l} {kv}: max err {err:.3e} x RMS > {max_tol} (worst {worst_max:.3e})"
        assert cos >= cos_tol, f"layer {l} {kv}: cosine {cos:.6f} < {cos_tol}"
        assert rc is None or rc >= resid_cos_tol, \
            f"layer {l} {kv}: residual cosine {rc:.6f} < {resid_cos_tol} (worst {worst_rc:.6f})"
    return worst_max, worst_cos, worst_rc, rows


def residual_cosine(got: np.ndarray, stale: np.ndarray, exact: np.ndarray, cache_dtype: str) -> float:
    """Cosine between the GPU's and the oracle's residual (repaired - stale)."""
    s = as_f64(stale) if cache_dtype == "bf16" else stale.astype(np.float64)
    g = (as_f64(got) if cache_dtype == "bf16" else got.astype(np.float64)) - s
    e = exact - s
    return float((g * e).sum() / np.sqrt((g ** 2).sum() * (e ** 2).sum()))
