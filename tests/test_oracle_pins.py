"""Pins for the oracle: checks against what the paper prints and what mathematics fixes.

None of these re-types the oracle's own formula.  They use the paper's printed
tables (tests/golden/), library routines that implement the textbook special
cases (torch SDPA, torch layer_norm/gelu, scipy block_diag), closed forms that
the method's definition implies, brute force on tiny inputs, and the
invariants the method's definition guarantees (Sec. 4.1).
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch
from scipy.linalg import block_diag

import fixtures as F
import oracle as O

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


# ------------------------------------------------------------------ paper tables
def _targets(golden):
    return {r[0]: tuple(int(x) for x in r[1:]) for r in golden("target_dims.txt")}


def _groups(tgt, db, B, ds, ratio=3):
    L, H, dh, dm = tgt
    return O.param_groups(n_layers=L, n_kv_heads=H, head_dim=dh, d_model=dm, d_seg=ds,
                          d_c=db, d_b=db, n_blocks=B, mlp_hidden=ratio * db)


def test_param_groups_match_paper_table(golden):
    """App. D Table repair-parameter-groups: every group and total, to one printed unit.

    The table prints millions to two decimals.  The oracle's shapes reproduce
    every entry to within 0.01 M; a wrong matrix shape (a transposed or
    missing projection, a gated MLP, a wrong D_KV) moves an entry by far more.
    """
    T = _targets(golden)
    for row in golden("param_groups.txt"):
        tgt, db, B, ds = row[0], int(row[1]), int(row[2]), int(row[3])
        enc, fus, rein, bb, head, other, total = map(float, row[4:])
        g = _groups(T[tgt], db, B, ds)
        got = {k: v / 1e6 for k, v in g.items()}
        assert other == 0.0
        for key, want in (("encoder", enc), ("fusion", fus), ("reinjection", rein),
                          ("backbone", bb), ("head", head), ("total", total)):
            assert abs(got[key] - want) <= 0.0101, (tgt, db, key, got[key], want)


def test_param_groups_reject_gated_mlp_and_ratio4(golden):
    """The same table rules out a ratio-4 MLP (the paper's repairers use ratio 3)."""
    T = _targets(golden)
    row = golden("param_groups.txt")[2]          # qwen2.5-3b, d_b 704
    g = _groups(T[row[0]], int(row[1]), int(row[2]), int(row[3]), ratio=4)
    assert abs(g["backbone"] / 1e6 - float(row[7])) > 1.0


def test_repair_scales_totals(golden):
    """App. A Table repair-scales: totals rounded to the nearest million."""
    T = _targets(golden)
    for tgt, size, db, B, ds, want in golden("repair_scales.txt"):
        g = _groups(T[tgt], int(db), int(B), int(ds))
        assert round(g["total"] / 1e6) == int(want), (tgt, size, g["total"])


def test_cache_payload_and_residual_width(golden):
    """App. I cache payload (2 N D_KV bytes) and App. D residual widths pin D_KV = 2 L H d_h."""
    T = _targets(golden)
    for tgt, n, mib in golden("cache_payload.txt"):
        L, H, dh, _ = T[tgt]
        assert O.cache_payload_bytes(int(n), L, H, dh) == int(mib) * 2 ** 20
    for tgt, dkv in golden("residual_width.txt"):
        L, H, dh, _ = T[tgt]
        shp = O.weight_shapes(n_layers=L, n_kv_heads=H, head_dim=dh, d_model=1, d_seg=1,
                              d_c=1, d_b=1, n_blocks=0, mlp_hidden=1)
        assert shp["head.w_out"][0] == int(dkv)


# ------------------------------------------------------------------ rounding
def _bf16_rne_fraction(x: float) -> float:
    """Brute-force RNE to bf16 with exact rational arithmetic."""
    fx = Fraction(x)
    if fx == 0:
        return 0.0
    sgn = -1 if fx < 0 else 1
    a = abs(fx)
    e = math.floor(math.log2(a))
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    ulp = Fraction(2) ** (e - 7)
    lo = (a // ulp) * ulp
    hi = lo + ulp
    if a - lo < hi - a:
        r = lo
    elif a - lo > hi - a:
        r = hi
    else:
        r = lo if (lo / ulp) % 2 == 0 else hi
    return float(sgn * r)


def test_round_to_cache_bf16_brute_force():
    g = np.random.default_rng(0)
    xs = list(g.normal(size=300) * 10 ** g.uniform(-3, 3, 300))
    # exact ties and near-ties that a double rounding through fp32 would get wrong
    for base in (1.0, 1.5, 3.25, 100.0, 0.0078125):
        ulp = 2.0 ** (math.floor(math.log2(base)) - 7)
        for frac in (0.5, 0.5 + 2 ** -30, 0.5 - 2 ** -30, 1.5, 0.25):
            xs += [base + frac * ulp, -(base + frac * ulp)]
    xs = np.asarray(xs, np.float64)
    got = O.dtype_to_f64(O.round_to_cache(xs, "bf16"), "bf16")
    want = np.asarray([_bf16_rne_fraction(float(x)) for x in xs])
    assert np.array_equal(got, want)
    f32 = g.normal(size=1000).astype(np.float32)
    t = torch.from_numpy(f32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.round_to_cache(f32.astype(np.float64), "bf16"), t)


# ------------------------------------------------------------------ textbook pieces
def test_layer_norm_and_gelu_match_torch():
    g = np.random.default_rng(1)
    x = g.normal(size=(37, 96)) * 3 + 1
    gam, bet = g.normal(size=96), g.normal(size=96)
    want = torch.nn.functional.layer_norm(torch.from_numpy(x), (96,), torch.from_numpy(gam),
                                          torch.from_numpy(bet), eps=1e-5).numpy()
    np.testing.assert_allclose(O.layer_norm(x, gam, bet, 1e-5), want, rtol=1e-12, atol=1e-12)
    want = torch.nn.functional.gelu(torch.from_numpy(x), approximate="none").numpy()
    np.testing.assert_allclose(O.gelu(x), want, rtol=1e-12, atol=1e-14)


def test_rope_is_complex_rotation():
    """Rotate-half RoPE == multiply (x_i + i x_{i+d/2}) by exp(i p f_i)."""
    g = np.random.default_rng(2)
    n, d = 11, 16
    x = g.normal(size=(n, 3, d))
    pos = g.integers(0, 5000, size=n)
    f = 10000.0 ** (-np.arange(d // 2) * 2.0 / d)
    got = O.rope_rotate_half(x, pos, f)
    z = (x[..., :d // 2] + 1j * x[..., d // 2:]) * np.exp(1j * pos[:, None, None] * f)
    np.testing.assert_allclose(got, np.concatenate([z.real, z.imag], -1), rtol=1e-10, atol=1e-10)
    np.testing.assert_array_equal(O.rope_rotate_half(x, np.zeros(n, int), f), x)
    back = O.rope_rotate_half(got, -pos, f)
    np.testing.assert_allclose(back, x, atol=1e-10)


def _sdpa(q, k, v, causal=False):
    # torch reference expects [heads, N, d]
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a.transpose(1, 0, 2)))
    o = torch.nn.functional.scaled_dot_product_attention(t(q), t(k), t(v), is_causal=causal)
    return o.numpy().transpose(1, 0, 2)


def test_attention_single_chunk_is_bidirectional_sdpa():
    g = np.random.default_rng(3)
    q, k, v = (g.normal(size=(50, 3, 8)) for _ in range(3))
    got = O.block_causal_attention(q, k, v, np.zeros(50, np.int32))
    np.testing.assert_allclose(got, _sdpa(q, k, v), rtol=1e-10, atol=1e-12)


def test_attention_unit_chunks_is_causal_sdpa():
    """All chunks of length 1: block-causal reduces to token-causal (ablation A1)."""
    g = np.random.default_rng(4)
    q, k, v = (g.normal(size=(40, 2, 16)) for _ in range(3))
    got = O.block_causal_attention(q, k, v, np.arange(40, dtype=np.int32))
    np.testing.assert_allclose(got, _sdpa(q, k, v, causal=True), rtol=1e-10, atol=1e-12)


def test_attention_brute_force_tiny():
    """Pure-Python loops over an explicit mask on a 7-token, 3-chunk input."""
    g = np.random.default_rng(5)
    cid = np.array([0, 0, 1, 1, 1, 2, 2], np.int32)
    n, nh, dh = 7, 2, 4
    q, k, v = (g.normal(size=(n, nh, dh)) for _ in range(3))
    want = np.zeros((n, nh, dh))
    for h in range(nh):
        for i in range(n):
            sc = []
            for j in range(n):
                if cid[j] <= cid[i]:
                    sc.append((j, sum(q[i, h, d] * k[j, h, d] for d in range(dh)) / math.sqrt(dh)))
            m = max(s for _, s in sc)
            den = sum(math.exp(s - m) for _, s in sc)
            for j, s in sc:
                for d in range(dh):
                    want[i, h, d] += math.exp(s - m) / den * v[j, h, d]
    np.testing.assert_allclose(O.block_causal_attention(q, k, v, cid), want, rtol=1e-12, atol=1e-13)


def test_attention_chunk_prefix_and_constant_values():
    g = np.random.default_rng(6)
    cid = np.array([0] * 9 + [1] * 5 + [2] * 7, np.int32)
    q, k, v = (g.normal(size=(21, 2, 8)) for _ in range(3))
    o = O.block_causal_attention(q, k, v, cid)
    # chunk 0 sees only itself: plain SDPA over the first 9 tokens
    np.testing.assert_allclose(o[:9], _sdpa(q[:9], k[:9], v[:9]), rtol=1e-10, atol=1e-12)
    # chunk 1 sees chunks 0 and 1 (rows of a 14-token bidirectional SDPA)
    np.testing.assert_allclose(o[9:14], _sdpa(q[:14], k[:14], v[:14])[9:], rtol=1e-10, atol=1e-12)
    # softmax weights sum to one: constant values pass through unchanged
    c = np.broadcast_to(g.normal(size=(1, 2, 8)), (21, 2, 8))
    np.testing.assert_allclose(O.block_causal_attention(q, k, c, cid), c, rtol=1e-12)


def test_stale_encoder_is_block_diagonal_product():
    """Per-segment linears == one product with block_diag(W_1..W_S) on kv / sigma."""
    c = F.make_case("tiny_affine")
    t, w = c.target, c.weights
    g = np.random.default_rng(7)
    kv = g.normal(size=(5, t.d_kv))
    W = O.dtype_to_f64(w["w_seg"], "bf16")
    BD = block_diag(*[W[s] for s in range(t.n_segments)])           # [S*d_seg, D_KV]
    y = (kv / w["sigma_stale"].astype(np.float64)) @ BD.T + w["b_seg"].reshape(-1)
    want = y @ O.dtype_to_f64(w["w_map"], "bf16").T + w["b_map"]
    got = O.stale_encoder(kv, w["sigma_stale"], w["w_seg"], w["b_seg"], w["w_map"], w["b_map"],
                          t.head_dim)
    np.testing.assert_allclose(got, want, rtol=1e-11, atol=1e-11)
    # dividing by sigma: scaling the cache and sigma together leaves s unchanged
    got2 = O.stale_encoder(kv * 4.0, w["sigma_stale"] * 4.0, w["w_seg"], w["b_seg"], w["w_map"],
                           w["b_map"], t.head_dim)
    np.testing.assert_allclose(got2, got, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------------ whole-method invariants
def _assembled(case):
    kvp, embp = case.pool()
    p = case.plan
    return O.assemble_stale(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)


def _run(case, a, w=None, **kw):
    t, r = case.target, case.repairer
    return O.repair_request(a["kv"], a["emb"], a["chunk_id"], a["pos"], w or case.weights,
                            cache_dtype=t.cache_dtype, n_layers=t.n_layers,
                            n_kv_heads=t.n_kv_heads, head_dim=t.head_dim, n_heads=r.n_heads,
                            **kw)


def test_assembly_is_the_chunk_concatenation():
    c = F.make_case("small_multi")
    kvp, embp = c.pool()
    a = _assembled(c)
    p = c.plan
    t = 0
    for r in range(len(p.cu_chunks) - 1):
        local = 0
        assert a["cu_seqlens"][r] == t
        for k, ch in enumerate(p.chunk_idx[p.cu_chunks[r]:p.cu_chunks[r + 1]]):
            for i in range(p.chunk_len[ch]):
                row = p.chunk_start[ch] + i
                assert np.array_equal(a["kv"][t], kvp[row]) and np.array_equal(a["emb"][t], embp[row])
                assert a["chunk_id"][t] == k and a["pos"][t] == local
                assert a["chunk_end"][t] == local - i + p.chunk_len[ch]
                t += 1
                local += 1
    assert a["cu_seqlens"][-1] == t == len(a["kv"])


@pytest.mark.parametrize("name", ["tiny", "small"])
def test_zero_head_returns_stale_bit_for_bit(name):
    """W_out = 0 and b_out = 0 (or sigma_Delta = 0): the repaired cache is the stale cache."""
    c = F.make_case(name)
    a = _assembled(c)
    for patch in ({"w_out": np.zeros_like(c.weights["w_out"]),
                   "b_out": np.zeros_like(c.weights["b_out"])},
                  {"sigma_delta": np.zeros_like(c.weights["sigma_delta"])}):
        w = dict(c.weights, **patch)
        res = _run(c, a, w)
        out = O.round_to_cache(res.repaired, c.target.cache_dtype)
        assert np.array_equal(out.view(np.uint8), np.ascontiguousarray(a["kv"]).view(np.uint8))


def test_causality_later_chunks_do_not_touch_earlier():
    """Perturbing chunks >= 2 leaves every output of chunks 0-1 bit-identical (A_ij)."""
    c = F.make_case("small")
    a = _assembled(c)
    res = _run(c, a)
    cut = int(np.searchsorted(a["chunk_id"], 2))
    b = dict(a)
    g = np.random.default_rng(8)
    b["kv"] = a["kv"].copy()
    b["emb"] = a["emb"].copy()
    b["kv"][cut:] = g.integers(0, 2 ** 14, size=b["kv"][cut:].shape).astype(np.uint16)
    b["emb"][cut:] = g.integers(0, 2 ** 14, size=b["emb"][cut:].shape).astype(np.uint16)
    res2 = _run(c, b)
    for x, y in ((res.s, res2.s), (res.h0, res2.h0), (res.yf, res2.yf), (res.repaired, res2.repaired)):
        assert np.array_equal(x[:cut], y[:cut])
        assert not np.allclose(x[cut:], y[cut:])
    for hb, hb2 in zip(res.blocks, res2.blocks):
        assert np.array_equal(hb[:cut], hb2[:cut])


def test_earlier_chunks_do_reach_later():
    """The mask is not block-diagonal: chunk 0 changes the outputs of chunk 1."""
    c = F.make_case("tiny")
    a = _assembled(c)
    res = _run(c, a)
    b = dict(a)
    b["kv"] = a["kv"].copy()
    b["kv"][:64] *= 1.5
    res2 = _run(c, b)
    assert not np.allclose(res.yf[64:], res2.yf[64:])


def test_permutation_within_chunk_permutes_outputs():
    """Permuting tokens (cache rows, embeddings and positions) inside a chunk permutes outputs."""
    c = F.make_case("small")
    a = _assembled(c)
    res = _run(c, a, inv_freq_target=c.inv_freq_target)
    lo = int(np.searchsorted(a["chunk_id"], 1))
    hi = int(np.searchsorted(a["chunk_id"], 2))
    perm = np.arange(len(a["kv"]))
    perm[lo:hi] = lo + np.random.default_rng(9).permutation(hi - lo)
    b = {k: (v[perm] if k in ("kv", "emb", "pos", "chunk_id", "chunk_end") else v)
         for k, v in a.items()}
    res2 = _run(c, b, inv_freq_target=c.inv_freq_target)
    for x, y in ((res.yf, res2.yf), (res.repaired, res2.repaired), (res.repaired_rot, res2.repaired_rot)):
        np.testing.assert_allclose(y, x[perm], rtol=1e-9, atol=1e-9 * np.abs(x).max())


def test_identity_blocks_leave_only_reinjection():
    """With every block's weights zero, each block is the identity on its input, so
    h^B = h^0 + sum_b P_b(s) and y_f = LN_f(h^B): a closed form of Sec. 4.1."""
    c = F.make_case("tiny_affine")
    a = _assembled(c)
    w = dict(c.weights)
    for b in range(c.repairer.n_blocks):
        for k in ("w_qkv", "b_qkv", "w_o", "b_o", "w_fc1", "b_fc1", "w_fc2", "b_fc2"):
            w[f"blk{b}.{k}"] = np.zeros_like(w[f"blk{b}.{k}"])
    res = _run(c, a, w)
    want = res.h0.copy()
    for b in range(c.repairer.n_blocks):
        want += res.s @ O.dtype_to_f64(w["w_rein"][b], "bf16").T + w["b_rein"][b]
    np.testing.assert_allclose(res.blocks[-1], want, rtol=1e-12, atol=1e-12)


def test_no_blocks_is_head_of_fused_input():
    c = F.make_case("tiny", repairer=F.RepairerDims(8, 64, 128, 0, 4, 512))
    a = _assembled(c)
    res = _run(c, a)
    want = torch.nn.functional.layer_norm(torch.from_numpy(res.h0), (128,), eps=1e-5).numpy()
    np.testing.assert_allclose(res.yf, want, rtol=1e-10, atol=1e-10)


def test_global_rope_properties():
    c = F.make_case("small")
    a = _assembled(c)
    res = _run(c, a, inv_freq_target=c.inv_freq_target)
    t = c.target
    n = len(a["kv"])
    rep = res.repaired.reshape(n, t.n_layers, 2, t.n_kv_heads, t.head_dim)
    rot = res.repaired_rot.reshape(n, t.n_layers, 2, t.n_kv_heads, t.head_dim)
    np.testing.assert_array_equal(rot[:, :, 1], rep[:, :, 1])           # V untouched
    np.testing.assert_array_equal(rot[0], rep[0])                       # p = 0: identity
    h = t.head_dim // 2
    nr = lambda x: x[..., :h] ** 2 + x[..., h:] ** 2
    np.testing.assert_allclose(nr(rot[:, :, 0]), nr(rep[:, :, 0]), rtol=1e-10)
    assert not np.allclose(rot[1:, :, 0], rep[1:, :, 0])


def test_constant_head_adds_sigma_times_bias():
    """W_out = 0, b_out = c: the head outputs c for every token, so the repaired cache
    is exactly KV_stale + sigma_Delta * c (Sec. 4.1 residual add, sign and scale)."""
    c = F.make_case("small")
    a = _assembled(c)
    g = np.random.default_rng(10)
    bias = g.normal(size=c.target.d_kv).astype(np.float32)
    w = dict(c.weights, w_out=np.zeros_like(c.weights["w_out"]), b_out=bias)
    res = _run(c, a, w)
    kv = O.dtype_to_f64(a["kv"], "bf16")
    want = kv + c.weights["sigma_delta"].astype(np.float64) * bias.astype(np.float64)
    np.testing.assert_array_equal(res.repaired, want)


# ------------------------------------------------------------------ whole method, brute force
def _lin(W, x, b):
    """Plain-Python affine map: out[i] = sum_k W[i][k] x[k] + b[i]."""
    return [sum(W[i][k] * x[k] for k in range(len(x))) + b[i] for i in range(len(W))]


def _ln(x, g, b, eps):
    n = len(x)
    mu = sum(x) / n
    var = sum((a - mu) ** 2 for a in x) / n
    return [(a - mu) / math.sqrt(var + eps) * g[i] + b[i] for i, a in enumerate(x)]


def _repair_brute_force(kv, emb, cid, pos, w, *, L, H, dh, n_heads, eps, theta):
    """The repair forward of Sec. 4.1 written out token by token with Python floats:
    StaleEncoder (one d_h -> d_seg map per segment on kv / sigma_stale, then W_map),
    token fusion F([s; P_tok e]), B pre-LN Repair Blocks whose input is h + P_b(s),
    each with rotate-half RoPE on q and k, softmax attention over keys j with
    c(j) <= c(i), an erf-GELU MLP, then LN_f, the head and kv + sigma_Delta z."""
    n, D = len(kv), len(kv[0])
    S = D // dh
    lst = lambda a: np.asarray(a, np.float64).tolist()
    sig = lst(w["sigma_stale"])
    s_feat = []
    for t in range(n):
        y = []
        for s in range(S):
            x = [kv[t][s * dh + d] / sig[s * dh + d] for d in range(dh)]
            y += _lin(lst(w["w_seg"][s]), x, lst(w["b_seg"][s]))
        s_feat.append(_lin(lst(w["w_map"]), y, lst(w["b_map"])))
    h = []
    for t in range(n):
        e = _lin(lst(w["w_tok"]), emb[t], lst(w["b_tok"]))
        h.append(_lin(lst(w["w_fuse"]), s_feat[t] + e, lst(w["b_fuse"])))
    db = len(h[0])
    hd = db // n_heads
    B = w["w_rein"].shape[0]
    for b in range(B):
        p = f"blk{b}."
        x = [[a + r for a, r in zip(h[t], _lin(lst(w["w_rein"][b]), s_feat[t], lst(w["b_rein"][b])))]
             for t in range(n)]
        q, k, v = [], [], []
        for t in range(n):
            u = _ln(x[t], lst(w[p + "ln1_g"]), lst(w[p + "ln1_b"]), eps)
            o = _lin(lst(w[p + "w_qkv"]), u, lst(w[p + "b_qkv"]))
            qt, kt = [], []
            for hh in range(n_heads):
                for src, dst in ((o[hh * hd:(hh + 1) * hd], qt), (o[db + hh * hd:db + (hh + 1) * hd], kt)):
                    half = hd // 2
                    for i in range(half):
                        ang = pos[t] * theta ** (-2.0 * i / hd)
                        c, sn = math.cos(ang), math.sin(ang)
                        dst.append(src[i] * c - src[i + half] * sn)
                    for i in range(half):
                        ang = pos[t] * theta ** (-2.0 * i / hd)
                        c, sn = math.cos(ang), math.sin(ang)
                        dst.append(src[i + half] * c + src[i] * sn)
            q.append(qt)
            k.append(kt)
            v.append(o[2 * db:])
        x2 = []
        for i in range(n):
            att = [0.0] * db
            for hh in range(n_heads):
                sl = slice(hh * hd, (hh + 1) * hd)
                sc = [(j, sum(a * c for a, c in zip(q[i][sl], k[j][sl])) / math.sqrt(hd))
                      for j in range(n) if cid[j] <= cid[i]]
                m = max(s for _, s in sc)
                den = sum(math.exp(s - m) for _, s in sc)
                for j, s in sc:
                    for d in range(hd):
                        att[hh * hd + d] += math.exp(s - m) / den * v[j][hh * hd + d]
            x2.append([a + c for a, c in zip(x[i], _lin(lst(w[p + "w_o"]), att, lst(w[p + "b_o"])))])
        h = []
        for t in range(n):
            u = _ln(x2[t], lst(w[p + "ln2_g"]), lst(w[p + "ln2_b"]), eps)
            g = [0.5 * a * (1.0 + math.erf(a / math.sqrt(2.0)))
                 for a in _lin(lst(w[p + "w_fc1"]), u, lst(w[p + "b_fc1"]))]
            h.append([a + c for a, c in zip(x2[t], _lin(lst(w[p + "w_fc2"]), g, lst(w[p + "b_fc2"])))])
    sd = lst(w["sigma_delta"])
    out = []
    for t in range(n):
        yf = _ln(h[t], lst(w["lnf_g"]), lst(w["lnf_b"]), eps)
        z = _lin(lst(w["w_out"]), yf, lst(w["b_out"]))
        out.append([kv[t][c] + sd[c] * z[c] for c in range(D)])
    return np.array(s_feat), np.array(out)


def test_whole_repair_brute_force_tiny():
    """The oracle's repair of a 7-token, 3-chunk request equals the token-by-token
    Python-float restatement of Sec. 4.1 (every weight, bias and LayerNorm affine
    random and nonzero, two blocks, two heads, two segments)."""
    g = np.random.default_rng(11)
    L, H, dh, dm = 1, 1, 4, 5          # D_KV = 2 L H d_h = 8: segments K and V of layer 0
    ds, dc, db, B, nh, hid = 2, 3, 4, 2, 2, 6
    S, D = 2 * L * H, 2 * L * H * dh
    r = lambda *shape: g.normal(size=shape) * 0.5
    w = {"w_seg": r(S, ds, dh), "b_seg": r(S, ds), "w_map": r(dc, S * ds), "b_map": r(dc),
         "w_tok": r(dc, dm), "b_tok": r(dc), "w_fuse": r(db, 2 * dc), "b_fuse": r(db),
         "w_rein": r(B, db, dc), "b_rein": r(B, db), "lnf_g": 1 + r(db), "lnf_b": r(db),
         "w_out": r(D, db), "b_out": r(D), "sigma_stale": 0.5 + g.random(D),
         "sigma_delta": 0.5 + g.random(D)}
    for b in range(B):
        p = f"blk{b}."
        w.update({p + "ln1_g": 1 + r(db), p + "ln1_b": r(db), p + "w_qkv": r(3 * db, db),
                  p + "b_qkv": r(3 * db), p + "w_o": r(db, db), p + "b_o": r(db),
                  p + "ln2_g": 1 + r(db), p + "ln2_b": r(db), p + "w_fc1": r(hid, db),
                  p + "b_fc1": r(hid), p + "w_fc2": r(db, hid), p + "b_fc2": r(db)})
    n = 7
    cid = np.array([0, 0, 1, 1, 1, 2, 2], np.int32)
    pos = np.arange(n)
    kv = g.normal(size=(n, D))
    emb = g.normal(size=(n, dm))
    eps, theta = 1e-5, 1e4
    res = O.repair_request(kv, emb, cid, pos, w, cache_dtype="f32", n_layers=L, n_kv_heads=H,
                           head_dim=dh, n_heads=nh, eps=eps, rope_theta=theta)
    s_bf, rep_bf = _repair_brute_force(kv.tolist(), emb.tolist(), cid.tolist(), pos.tolist(), w, L=L,
                                       H=H, dh=dh, n_heads=nh, eps=eps, theta=theta)
    np.testing.assert_allclose(res.s, s_bf, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(res.repaired, rep_bf, rtol=1e-10, atol=1e-11)
    # and the restatement is sensitive to what it checks: V and K swapped in the
    # qkv split, or the mask reversed, move the result well outside the tolerance
    w_sw = dict(w)
    for b in range(B):
        q_, k_, v_ = np.split(w[f"blk{b}.w_qkv"], 3)
        w_sw[f"blk{b}.w_qkv"] = np.concatenate([q_, v_, k_])
    res_sw = O.repair_request(kv, emb, cid, pos, w_sw, cache_dtype="f32", n_layers=L, n_kv_heads=H,
                              head_dim=dh, n_heads=nh, eps=eps, rope_theta=theta)
    assert np.abs(res_sw.repaired - rep_bf).max() > 1e-3
