"""Pins for the oracle's mask and output variants (App. F, Sec. 2.2).

As in test_oracle_pins.py, nothing here re-types the oracle's formula: the
masks are checked against their library forms (numpy tril, scipy block_diag),
the masked attention against torch SDPA (with and without a boolean mask),
per-chunk SDPA and brute force, and the whole-network variants against the
invariants each mask implies and closed forms of the output choices.
"""
import math

import numpy as np
import pytest
import torch
from scipy.linalg import block_diag

import fixtures as F
import oracle as O

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")

CID = np.array([0] * 5 + [1] * 3 + [2] * 1 + [3] * 7, np.int32)     # 16 tokens, 4 chunks


def _sdpa(q, k, v, causal=False, mask=None):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.transpose(1, 0, 2)))
    m = None if mask is None else torch.from_numpy(mask)
    o = torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v), attn_mask=m, is_causal=causal)
    return o.numpy().transpose(1, 0, 2)


def _qkv(seed, n, nh=2, dh=8):
    g = np.random.default_rng(seed)
    return tuple(g.normal(size=(n, nh, dh)) for _ in range(3))


# ------------------------------------------------------------------ masks
def test_masks_match_library_forms():
    n = len(CID)
    lens = np.bincount(CID)
    assert np.array_equal(O.attention_mask(CID, "block_causal"), O.block_causal_mask(CID))
    assert np.array_equal(O.attention_mask(CID, "token_causal"), np.tril(np.ones((n, n), bool)))
    assert np.array_equal(O.attention_mask(CID, "bidirectional"), np.ones((n, n), bool))
    bd = block_diag(*[np.ones((m, m)) for m in lens]).astype(bool)
    assert np.array_equal(O.attention_mask(CID, "block_diagonal"), bd)
    # A3 is the symmetric part of A0: c(j) <= c(i) and c(i) <= c(j)
    a0 = O.attention_mask(CID, "block_causal")
    assert np.array_equal(O.attention_mask(CID, "block_diagonal"), a0 & a0.T)
    with pytest.raises(ValueError):
        O.attention_mask(CID, "sliding")


def test_masked_attention_special_cases_are_sdpa():
    q, k, v = _qkv(21, len(CID))
    m = lambda mode: O.attention_mask(CID, mode)
    np.testing.assert_allclose(O.masked_attention(q, k, v, m("bidirectional")), _sdpa(q, k, v),
                               rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(O.masked_attention(q, k, v, m("token_causal")), _sdpa(q, k, v, causal=True),
                               rtol=1e-10, atol=1e-12)
    # block-diagonal: each chunk is an independent bidirectional SDPA
    want = np.concatenate([_sdpa(q[CID == c], k[CID == c], v[CID == c]) for c in np.unique(CID)])
    np.testing.assert_allclose(O.masked_attention(q, k, v, m("block_diagonal")), want, rtol=1e-10, atol=1e-12)
    # the method's mask through the generic path equals the chunk-prefix form
    np.testing.assert_allclose(O.masked_attention(q, k, v, m("block_causal")),
                               O.block_causal_attention(q, k, v, CID), rtol=1e-10, atol=1e-12)


def test_masked_attention_arbitrary_mask_is_sdpa():
    g = np.random.default_rng(22)
    n = 23
    q, k, v = _qkv(23, n, nh=3, dh=4)
    mask = g.random((n, n)) < 0.3
    mask[np.arange(n), g.integers(0, n, size=n)] = True          # every row sees something
    np.testing.assert_allclose(O.masked_attention(q, k, v, mask), _sdpa(q, k, v, mask=mask),
                               rtol=1e-10, atol=1e-12)


def test_masked_attention_brute_force_tiny():
    q, k, v = _qkv(24, 6, nh=1, dh=3)
    mask = np.array([[1, 0, 0, 1, 0, 0], [1, 1, 0, 0, 0, 0], [0, 0, 1, 0, 0, 0],
                     [1, 1, 1, 1, 1, 1], [0, 0, 0, 0, 1, 1], [0, 1, 0, 1, 0, 1]], bool)
    want = np.zeros_like(q)
    for i in range(6):
        vis = [j for j in range(6) if mask[i, j]]
        sc = [sum(q[i, 0, d] * k[j, 0, d] for d in range(3)) / math.sqrt(3) for j in vis]
        mx = max(sc)
        den = sum(math.exp(s - mx) for s in sc)
        for j, s in zip(vis, sc):
            want[i, 0] += math.exp(s - mx) / den * v[j, 0]
    np.testing.assert_allclose(O.masked_attention(q, k, v, mask), want, rtol=1e-12, atol=1e-13)


def test_block_diagonal_unit_chunks_return_values_exactly():
    """A3 with one-token chunks: each query sees only itself, softmax weight 1."""
    q, k, v = _qkv(25, 9)
    out = O.masked_attention(q, k, v, O.attention_mask(np.arange(9, dtype=np.int32), "block_diagonal"))
    assert np.array_equal(out, v)


# ------------------------------------------------------------------ whole network under each mask
def _assembled(case):
    kvp, embp = case.pool()
    p = case.plan
    return O.assemble_stale(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)


def _run(case, a, w=None, **kw):
    t, r = case.target, case.repairer
    return O.repair_request(a["kv"], a["emb"], a["chunk_id"], a["pos"], w or case.weights,
                            cache_dtype=t.cache_dtype, n_layers=t.n_layers,
                            n_kv_heads=t.n_kv_heads, head_dim=t.head_dim, n_heads=r.n_heads, **kw)


def _perturb(a, rows, seed):
    g = np.random.default_rng(seed)
    b = dict(a)
    b["kv"], b["emb"] = a["kv"].copy(), a["emb"].copy()
    b["kv"][rows] = g.integers(0, 2 ** 14, size=b["kv"][rows].shape).astype(np.uint16)
    b["emb"][rows] = g.integers(0, 2 ** 14, size=b["emb"][rows].shape).astype(np.uint16)
    return b


def _same_rows(r1, r2, rows):
    return all(np.array_equal(x[rows], y[rows]) for x, y in
               ((r1.yf, r2.yf), (r1.repaired, r2.repaired)))


@pytest.fixture(scope="module")
def tiny_small():
    c = F.make_case("tiny")
    return c, _assembled(c)


def test_block_diagonal_chunks_are_independent(tiny_small):
    """A3: changing chunk 1 leaves every output of chunk 0 bit-identical, and vice versa."""
    c, a = tiny_small
    cid = a["chunk_id"]
    base = _run(c, a, mask_mode="block_diagonal")
    for ch in (0, 1):
        rows = cid == ch
        other = ~rows
        r2 = _run(c, _perturb(a, rows, 30 + ch), mask_mode="block_diagonal")
        assert _same_rows(base, r2, other)
        assert not np.allclose(base.yf[rows], r2.yf[rows])
    # ... while under A0 chunk 0 does reach chunk 1
    r0 = _run(c, a)
    r0b = _run(c, _perturb(a, cid == 0, 30))
    assert not np.allclose(r0.yf[cid == 1], r0b.yf[cid == 1])


def test_token_causal_prefix_is_independent_of_suffix(tiny_small):
    """A1: changing tokens >= t (t inside chunk 0) leaves tokens < t bit-identical."""
    c, a = tiny_small
    t = 37
    rows = np.arange(len(a["kv"])) >= t
    base = _run(c, a, mask_mode="token_causal")
    r2 = _run(c, _perturb(a, rows, 31), mask_mode="token_causal")
    assert _same_rows(base, r2, ~rows)
    assert not np.allclose(base.yf[rows], r2.yf[rows])
    # under A0 the same change does reach token 0 (same chunk)
    r0, r0b = _run(c, a), _run(c, _perturb(a, rows, 31))
    assert not np.allclose(r0.yf[:1], r0b.yf[:1])


def test_bidirectional_later_chunks_reach_earlier(tiny_small):
    """A2: the last chunk changes the first chunk's outputs (A0 would not)."""
    c, a = tiny_small
    cid = a["chunk_id"]
    last = cid == cid.max()
    base = _run(c, a, mask_mode="bidirectional")
    r2 = _run(c, _perturb(a, last, 32), mask_mode="bidirectional")
    assert not np.allclose(base.yf[cid == 0], r2.yf[cid == 0])
    r0, r0b = _run(c, a), _run(c, _perturb(a, last, 32))
    assert _same_rows(r0, r0b, cid == 0)


def test_single_chunk_masks_agree():
    """One chunk: A0, A2 and A3 are all the full bidirectional mask."""
    c = F.make_case("tiny", requests=[[0]], n_req_chunks=None)
    a = _assembled(c)
    ref = _run(c, a)
    for mode in ("bidirectional", "block_diagonal"):
        np.testing.assert_allclose(_run(c, a, mask_mode=mode).repaired, ref.repaired,
                                   rtol=1e-11, atol=1e-11)


# ------------------------------------------------------------------ output choices
def _dims(c):
    t = c.target
    return dict(n_layers=t.n_layers, n_kv_heads=t.n_kv_heads, head_dim=t.head_dim)


def test_component_columns_follow_coordinate_order():
    """K and V alternate in blocks of H*d_h per layer, K first (R9): brute force."""
    L, H, dh = 3, 2, 4
    k = O.component_columns("k", n_layers=L, n_kv_heads=H, head_dim=dh)
    v = O.component_columns("v", n_layers=L, n_kv_heads=H, head_dim=dh)
    want_k = []
    for layer in range(L):
        for kind in range(2):
            want_k += [kind == 0] * (H * dh)
    assert np.array_equal(k, np.array(want_k)) and np.array_equal(v, ~k)
    assert O.component_columns("kv", n_layers=L, n_kv_heads=H, head_dim=dh).all()


def test_output_choices_partition_the_full_repair(tiny_small):
    c, a = tiny_small
    res = _run(c, a)
    kw = dict(cache_dtype=c.target.cache_dtype, **_dims(c))
    sd = c.weights["sigma_delta"]
    full = O.apply_output_choice(a["kv"], res.z, sd, **kw)
    assert np.array_equal(full, res.repaired)             # same as the method's residual add
    ko = O.apply_output_choice(a["kv"], res.z, sd, component="k", **kw)
    vo = O.apply_output_choice(a["kv"], res.z, sd, component="v", **kw)
    kc = O.component_columns("k", **_dims(c))
    stale = O.dtype_to_f64(a["kv"], c.target.cache_dtype)
    assert np.array_equal(ko[:, kc], full[:, kc]) and np.array_equal(ko[:, ~kc], stale[:, ~kc])
    assert np.array_equal(vo[:, ~kc], full[:, ~kc]) and np.array_equal(vo[:, kc], stale[:, kc])
    keep = a["chunk_id"] == 0
    kf = O.apply_output_choice(a["kv"], res.z, sd, keep_rows=keep, **kw)
    assert np.array_equal(kf[keep], stale[keep]) and np.array_equal(kf[~keep], full[~keep])


def test_zero_offset_constant_head_closed_form(tiny_small):
    """A5 with W_out = 0, b_out = c: every token's output is sigma_Delta * c, whatever the stale cache."""
    c, a = tiny_small
    g = np.random.default_rng(33)
    bias = g.normal(size=c.target.d_kv).astype(np.float32)
    w = dict(c.weights, w_out=np.zeros_like(c.weights["w_out"]), b_out=bias)
    res = _run(c, a, w)
    out = O.apply_output_choice(a["kv"], res.z, c.weights["sigma_delta"], offset="zero",
                                cache_dtype=c.target.cache_dtype, **_dims(c))
    want = c.weights["sigma_delta"].astype(np.float64) * bias.astype(np.float64)
    assert np.array_equal(out, np.broadcast_to(want, out.shape))


def test_stale_kv_cache_inverts_canonicalisation():
    """R_M(p) on the canonical K, then R_M(p)^{-1} (the offline canonicalisation), returns it."""
    c = F.make_case("small")
    a = _assembled(c)
    kw = dict(cache_dtype=c.target.cache_dtype, **_dims(c))
    st = O.stale_kv_cache_exact(a["kv"], a["pos"], c.inv_freq_target, **kw)
    back = O.canonical_exact(st, a["pos"], c.inv_freq_target, n_layers=c.target.n_layers,
                             n_kv_heads=c.target.n_kv_heads, head_dim=c.target.head_dim,
                             cache_dtype="f32")          # float64 values pass through exactly
    np.testing.assert_allclose(back, O.dtype_to_f64(a["kv"], "bf16"), rtol=0, atol=1e-9)


def test_stale_kv_cache_is_complex_rotation_of_k():
    c = F.make_case("small")
    a = _assembled(c)
    t = c.target
    n = len(a["kv"])
    st = O.stale_kv_cache_exact(a["kv"], a["pos"], c.inv_freq_target, cache_dtype="bf16", **_dims(c))
    x = O.dtype_to_f64(a["kv"], "bf16").reshape(n, t.n_layers, 2, t.n_kv_heads, t.head_dim)
    y = st.reshape(x.shape)
    h = t.head_dim // 2
    f = c.inv_freq_target.astype(np.float64)
    zc = (x[:, :, 0, :, :h] + 1j * x[:, :, 0, :, h:]) * np.exp(1j * a["pos"][:, None, None, None] * f)
    np.testing.assert_allclose(y[:, :, 0, :, :h], zc.real, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(y[:, :, 0, :, h:], zc.imag, rtol=1e-12, atol=1e-12)
    assert np.array_equal(y[:, :, 1], x[:, :, 1])                 # V as stored
    assert np.array_equal(y[a["pos"] == 0], x[a["pos"] == 0])      # p = 0: identity


def test_output_choice_with_target_rope_rotates_every_k(tiny_small):
    """R19: V-only repair still leaves K rotated (the stale cache's K), V repaired."""
    c, a = tiny_small
    res = _run(c, a)
    kw = dict(cache_dtype=c.target.cache_dtype, **_dims(c))
    vo = O.apply_output_choice(a["kv"], res.z, c.weights["sigma_delta"], component="v",
                               pos=a["pos"], inv_freq_target=c.inv_freq_target, **kw)
    st = O.stale_kv_cache_exact(a["kv"], a["pos"], c.inv_freq_target, **kw)
    kc = O.component_columns("k", **_dims(c))
    full = O.apply_output_choice(a["kv"], res.z, c.weights["sigma_delta"], **kw)
    assert np.array_equal(vo[:, kc], st[:, kc])
    assert np.array_equal(vo[:, ~kc], full[:, ~kc])
