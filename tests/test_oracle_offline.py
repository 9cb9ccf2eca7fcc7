"""Pins of the offline oracle (chunk canonicalisation, sigma statistics) against
facts fixed by the paper and by the mathematics, independent of its code."""
import math

import numpy as np

import fixtures as F
import oracle as O


def _bf16(x):
    return F.f32_to_bf16(np.asarray(x, np.float32))


def test_canonical_worked_example():
    # one layer, one head, d_h = 4: pairs (0, 2) and (1, 3) with frequencies 1 and 1/2.
    # R_M(q)^{-1} rotates each pair by -q f: (a, b) -> (a cos + b sin, b cos - a sin).
    q = math.pi / 2
    kv = np.array([[1.0, 0.0, 0.0, 2.0, 5.0, 6.0, 7.0, 8.0]], np.float32)   # K then V
    out = O.canonical_exact(kv, np.array([q]), np.array([1.0, 0.5], np.float32), n_layers=1,
                            n_kv_heads=1, head_dim=4, cache_dtype="f32")
    c, s = math.cos(q / 2), math.sin(q / 2)
    want = [0.0, 2.0 * s, -1.0, 2.0 * c, 5.0, 6.0, 7.0, 8.0]
    np.testing.assert_allclose(out[0], want, atol=1e-15)


def _cache(n, L=2, H=2, dh=8, seed=0):
    g = np.random.default_rng(seed)
    return _bf16(g.standard_normal((n, 2 * L * H * dh))), dict(n_layers=L, n_kv_heads=H, head_dim=dh)


def test_canonical_position_zero_is_identity_and_v_untouched():
    kv, dims = _cache(7)
    inv = (1e4 ** (-np.arange(0, 8, 2) / 8)).astype(np.float32)
    out = O.canonicalize_chunk(kv, np.zeros(7, np.int32), inv, cache_dtype="bf16", **dims)
    assert np.array_equal(out, kv)
    pos = np.arange(7, dtype=np.int32) * 37
    out = O.canonicalize_chunk(kv, pos, inv, cache_dtype="bf16", **dims)
    v = lambda a: a.reshape(7, 2, 2, 2, 8)[:, :, 1]
    assert np.array_equal(v(out), v(kv))                      # V is stored as it is


def test_canonical_inverts_the_target_rope_and_keeps_pair_norms():
    kv, dims = _cache(9, seed=1)
    inv = (5e5 ** (-np.arange(0, 8, 2) / 8)).astype(np.float32)
    pos = np.arange(9, dtype=np.int32) * 101
    canon = O.canonical_exact(kv, pos, inv, cache_dtype="bf16", **dims)
    back = O.global_rope_k(canon, pos, inv, dims["n_layers"], dims["n_kv_heads"], dims["head_dim"])
    np.testing.assert_allclose(back, O.dtype_to_f64(kv, "bf16"), rtol=0, atol=1e-12)
    k = lambda a: a.reshape(9, 2, 2, 2, 8)[:, :, 0]
    x, y = k(O.dtype_to_f64(kv, "bf16")), k(canon)
    nx = x[..., :4] ** 2 + x[..., 4:] ** 2
    ny = y[..., :4] ** 2 + y[..., 4:] ** 2
    np.testing.assert_allclose(ny, nx, rtol=1e-13)


def test_sigma_rms_closed_forms():
    # a constant column c has RMS |c|; a column of +-a has RMS a
    a = np.zeros((6, 4), np.float32)
    a[:, 0] = 3.0
    a[:, 1] = [2, -2, 2, -2, 2, -2]
    a[:, 2] = -0.5
    r = O.sigma_rms([a], "f32")
    np.testing.assert_allclose(r, [3.0, 2.0, 0.5, 0.0])
    # pooling caches = concatenating them; a difference with itself is zero
    b = np.arange(12, dtype=np.float32).reshape(3, 4)
    np.testing.assert_allclose(O.sigma_rms([a, b], "f32"), O.sigma_rms([np.concatenate([a, b])], "f32"))
    assert np.all(O.sigma_rms([b], "f32", minus=[b]) == 0)
    # brute force on a tiny bf16 case
    kv, _ = _cache(5, seed=2)
    x = O.dtype_to_f64(kv, "bf16")
    brute = [math.sqrt(sum(x[t, j] ** 2 for t in range(5)) / 5) for j in range(x.shape[1])]
    np.testing.assert_allclose(O.sigma_rms([kv], "bf16"), brute, rtol=1e-14)
