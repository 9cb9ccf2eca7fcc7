"""Each kernel of the repair path against the oracle's step, through the C ABI."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import build, cr
from parity_util import as_f64, assert_close, assert_close_bf16, to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    L = cr.lib()
    cr.cr_clear_device_status()
    yield L
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, f"device status {word}"


def _bf16(g, shape, scale=1.0):
    return F.f32_to_bf16((g.standard_normal(shape) * scale).astype(np.float32))


# the last two shapes make the launcher pick 160-wide (fp32 residual add) and
# 192-wide (bf16, GELU) tiles with a ragged last column tile
@pytest.mark.parametrize("M,N,K", [(128, 128, 64), (300, 256, 200), (77, 3072, 1024),
                                   (513, 1024, 4096), (40, 48, 8), (1000, 512, 8192),
                                   (5120, 1008, 320), (5120, 528, 640)])
@pytest.mark.parametrize("epi", [cr.CR_EPI_BF16, cr.CR_EPI_GELU_BF16, cr.CR_EPI_ADD_F32, cr.CR_EPI_F32])
def test_linear(M, N, K, epi):
    g = np.random.default_rng(M * 7 + N + K + epi)
    A = _bf16(g, (M, K))
    W = _bf16(g, (N, K), 1.0 / np.sqrt(K))
    bias = g.standard_normal(N).astype(np.float32)
    ref = as_f64(A) @ as_f64(W).T + bias
    f32 = epi in (cr.CR_EPI_ADD_F32, cr.CR_EPI_F32)
    init = g.standard_normal((M, N)).astype(np.float32)
    out = to_dev(init) if f32 else torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    cr.cr_linear(to_dev(A), to_dev(W), to_dev(bias), out, epi)
    torch.cuda.synchronize()
    got = to_host(out)
    if epi == cr.CR_EPI_GELU_BF16:
        ref = O.gelu(ref)
    if epi == cr.CR_EPI_ADD_F32:
        ref = ref + init
    if f32:
        assert_close(got, ref, 1e-5, 1e-4, f"linear f32 {M}x{N}x{K}")
    else:   # one bf16 rounding of the output
        assert_close_bf16(got, ref, 3e-3, f"linear bf16 {M}x{N}x{K}")


@pytest.mark.parametrize("M,N,K", [(256, 128, 64), (300, 192, 1000), (1024, 4096, 5120), (16384, 1024, 336),
                                   (5120, 512, 2048), (128, 64, 8), (256, 128, 16384)])
@pytest.mark.parametrize("a_trans", [False, True])
@pytest.mark.parametrize("accumulate", [False, True])
def test_matmul_layouts(M, N, K, a_trans, accumulate):
    """The backward's products: C (+)= op(A) B with B stored [K, N] and A stored
    [M, K] or [K, M] (the MN-major operand layouts), against float64 products of
    the same bf16 values: fp32 accumulation error only.  Ragged K and M (not a
    multiple of the tile) included."""
    if a_trans and M % 64:
        pytest.skip("a transposed A needs whole 64-row blocks")
    g = np.random.default_rng(M + 3 * N + 7 * K + 2 * a_trans + accumulate)
    A = _bf16(g, (K, M) if a_trans else (M, K))
    B = _bf16(g, (K, N), 1.0 / np.sqrt(K))
    init = g.standard_normal((M, N)).astype(np.float32)
    C = to_dev(init)
    cr.cr_matmul(to_dev(A), to_dev(B), C, a_trans=a_trans, accumulate=accumulate)
    torch.cuda.synchronize()
    a64 = as_f64(A).T if a_trans else as_f64(A)
    ref = a64 @ as_f64(B) + (init if accumulate else 0.0)
    # fp32 accumulation: the error grows with the k-loop (measured 1.9e-5 relative RMS
    # at K = 16384); 1.5x that growth beyond K = 8192
    g = max(1.0, 1.5 * K / 8192)
    tol = (1e-5 * g, 1e-4 * g)
    assert_close(to_host(C), ref, *tol, f"matmul {M}x{N}x{K} a_trans={a_trans} acc={accumulate}")
    # with a workspace the poorly filled shapes with long k-loops (the last one here)
    # run as k-parts summed in order: the same products to fp32 rounding, and the
    # same bits on a rerun
    ws = torch.empty(8 * M * N * 4, dtype=torch.uint8, device="cuda")
    outs = []
    for _ in range(2):
        C2 = to_dev(init)
        cr.cr_matmul(to_dev(A), to_dev(B), C2, a_trans=a_trans, accumulate=accumulate, workspace=ws)
        torch.cuda.synchronize()
        outs.append(to_host(C2))
    assert_close(outs[0], ref, *tol, f"split matmul {M}x{N}x{K} a_trans={a_trans} acc={accumulate}")
    assert np.array_equal(outs[0], outs[1])


def test_gelu_epilogue_tails():
    """GELU of the GEMM epilogue over [-12, 12]: every row's output equals x, so
    the epilogue sees each bf16 value of the range; compared with the fp64
    definition x/2 erfc(-x / sqrt 2) (= x/2 (1 + erf(x / sqrt 2)) without the
    tail cancellation).  The epilogue's GELU is accurate to 1e-7 absolute and to
    1.5e-3 relative wherever |GELU| >= 5e-5 (x >= -4.2), so those outputs are one
    bf16 rounding of the exact value; the smaller outputs of the far negative tail
    are held to the absolute bound."""
    sp = pytest.importorskip("scipy.special")
    M, K, N = 4096, 16, 16
    x = F.f32_to_bf16(np.linspace(-12.0, 12.0, M).astype(np.float32))
    A = np.zeros((M, K), np.uint16)
    A[:, 0] = x
    W = np.zeros((N, K), np.uint16)
    W[:, 0] = F.f32_to_bf16(np.ones(N, np.float32))
    out = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    cr.cr_linear(to_dev(A), to_dev(W), to_dev(np.zeros(N, np.float32)), out, cr.CR_EPI_GELU_BF16)
    torch.cuda.synchronize()
    got = as_f64(to_host(out))
    xf = as_f64(x)
    ref = (0.5 * xf * sp.erfc(-xf / np.sqrt(2.0)))[:, None] * np.ones((1, N))
    # one bf16 rounding (half an ulp, 2^-9 relative) plus float32 evaluation error
    err = np.abs(got - ref)
    big = np.abs(ref) >= 5e-5
    assert np.all(err[big] <= 2.0 ** -8 * np.abs(ref[big])), float(np.max(err[big] / np.abs(ref[big])))
    assert np.all(err <= 1e-7 + 2.0 ** -8 * np.abs(ref)), float(np.max(err))
    assert np.all(got[xf > 0] > 0) and np.all(got[xf < 0] <= 0)   # sign of x, never above 0 for x < 0


@pytest.mark.parametrize("D", [128, 512, 1024])
def test_layernorm_with_reinjection_add(D):
    g = np.random.default_rng(D)
    M = 301
    x = (g.standard_normal((M, D)) * 3 + 0.5).astype(np.float32)
    add = g.standard_normal((M, 2 * D)).astype(np.float32)   # strided slice, like P_b(s)
    gam = (1 + 0.2 * g.standard_normal(D)).astype(np.float32)
    bet = (0.1 * g.standard_normal(D)).astype(np.float32)
    xd = to_dev(x)
    xo = torch.empty_like(xd)
    u = torch.empty(M, D, dtype=torch.bfloat16, device="cuda")
    addd = to_dev(add)
    cr.cr_layernorm(xd, to_dev(gam), to_dev(bet), 1e-5, u, add=addd[:, D:], ld_add=2 * D, x_out=xo)
    torch.cuda.synchronize()
    xs = x.astype(np.float64) + as_f64(add)[:, D:]
    np.testing.assert_allclose(to_host(xo), xs, rtol=1e-6, atol=1e-6)
    assert_close_bf16(to_host(u), O.layer_norm(xs, gam, bet, 1e-5), 3e-3, "layernorm")


def _chunk_ids(lens):
    return np.concatenate([np.full(n, i, np.int32) for i, n in enumerate(lens)])


def _attention_check(reqs, hd, nh, seed, what):
    """cr_chunk_causal_attention on random bf16 Q, K, V for requests of the given
    chunk lengths, every output against the oracle's block-causal attention."""
    g = np.random.default_rng(seed)
    db = nh * hd
    lens = [int(sum(r)) for r in reqs]
    N = sum(lens)
    qkv = _bf16(g, (N, 3 * db))
    cend = []
    for r in reqs:
        e = np.cumsum(r)
        cend.append(np.concatenate([np.full(n, e[i], np.int32) for i, n in enumerate(r)]))
    cend = np.concatenate(cend)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    out = torch.full((N, db), float("nan"), dtype=torch.bfloat16, device="cuda")
    cr.cr_chunk_causal_attention(to_dev(qkv), db, nh, to_dev(cend), cu, out)
    torch.cuda.synchronize()
    got = to_host(out)
    q = as_f64(qkv)
    want = np.empty((N, db))
    mag = np.empty((N, db))
    for r, req in enumerate(reqs):
        a, b = cu[r], cu[r + 1]
        sl = lambda off: q[a:b, off:off + db].reshape(b - a, nh, hd)
        cid = _chunk_ids(req)
        want[a:b] = O.block_causal_attention(sl(0), sl(db), sl(2 * db), cid).reshape(b - a, db)
        # sum_j p_j |v_j| / sum_j p_j: the scale of each output's P-rounding error
        mag[a:b] = O.block_causal_attention(sl(0), sl(db), np.abs(sl(2 * db)), cid).reshape(b - a, db)
    g = as_f64(got)
    assert not np.isnan(g).any()
    # P enters the PV product rounded to bf16 (relative error <= 2^-9 per weight) and
    # the output is rounded once to bf16: |err| <= 2^-9 mag + 2^-9 |o|; 2x margin.
    bound = 2.0 ** -8 * mag + 2.0 ** -8 * np.abs(want) + 1e-5
    worst = float((np.abs(g - want) / bound).max())
    print(f"attention {what}: N {N}, error / bound = {worst:.3f}")
    assert worst <= 1.0, f"attention {what}: error / bound = {worst:.3f}"
    assert_close(got, want, 8e-3, 1.0, f"attention {what}")


@pytest.mark.parametrize("hd", [32, 64])
@pytest.mark.parametrize("reqs", [
    [[64, 64]],                      # two chunks, one tile
    [[300]],                          # single chunk: bidirectional, ragged tail
    [[1] * 150],                      # unit chunks: token-causal
    [[130, 77, 200, 1, 95]],          # ragged chunk map across several tiles
    [[129, 40], [5], [300, 256, 3]],  # several requests (varlen)
])
def test_chunk_causal_attention(hd, reqs):
    _attention_check(reqs, hd, 4 if hd == 32 else 8, hd + sum(map(sum, reqs)), f"hd={hd} {reqs}")


@pytest.mark.slow
@pytest.mark.parametrize("name", ["llama8b", "qwen7b"])
def test_chunk_causal_attention_full_size(name):
    """A whole request of a workload, every row checked: the 8B shape's 5120 tokens
    in ten 512-token chunks (20 query-tile pairs per head, many passes around the
    kernel's K/V ring) and the 7B shape's ragged 20-chunk map (chunk ends inside
    tiles), both with the workloads' 16 heads of 64."""
    c = F.make_case(name)
    p = c.plan
    lens = [int(x) for x in p.chunk_len[p.chunk_idx[p.cu_chunks[0]:p.cu_chunks[1]]]]
    _attention_check([lens], c.repairer.head_dim, c.repairer.n_heads, 17, name)


@pytest.mark.parametrize("db,nh", [(128, 4), (512, 8), (1024, 16)])
def test_qkv_rope(db, nh):
    g = np.random.default_rng(db)
    N = 333
    u = _bf16(g, (N, db))
    W = _bf16(g, (3 * db, db), 1 / np.sqrt(db))
    b = (0.1 * g.standard_normal(3 * db)).astype(np.float32)
    pos = g.integers(0, 9000, N).astype(np.int32)
    out = torch.empty(N, 3 * db, dtype=torch.bfloat16, device="cuda")
    cr.cr_qkv_rope(to_dev(u), to_dev(W), to_dev(b), to_dev(pos), db, nh, 1e4, out)
    torch.cuda.synchronize()
    hd = db // nh
    y = as_f64(u) @ as_f64(W).T + b
    f = O.repair_inv_freq(hd, 1e4)
    q = O.rope_rotate_half(y[:, :db].reshape(N, nh, hd), pos, f).reshape(N, db)
    k = O.rope_rotate_half(y[:, db:2 * db].reshape(N, nh, hd), pos, f).reshape(N, db)
    want = np.concatenate([q, k, y[:, 2 * db:]], axis=1)
    assert_close(to_host(out), want, 4e-3, 2e-2, "qkv+rope")


@pytest.mark.parametrize("name", ["tiny", "small", "llama8b"])
def test_segment_projection(name):
    c = F.make_case(name)
    t, r = c.target, c.repairer
    rows = 300 if name != "llama8b" else 1000
    kv, _ = c.pool_rows(0, rows)
    if t.cache_dtype == "f32":
        kv = F.f32_to_bf16(kv)          # the op consumes bf16 (fp32 caches are converted first)
    w = c.weights
    from paper_2609_35139_gb300 import dims_from
    td, _ = dims_from(t, r)
    y = torch.empty(rows, t.n_segments * r.d_seg, dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(t.n_segments * r.d_seg * t.head_dim * 4, dtype=torch.uint8, device="cuda")
    cr.cr_segment_project(td, r.d_seg, to_dev(kv), to_dev(w["w_seg"]), to_dev(w["b_seg"]),
                          to_dev(w["sigma_stale"]), y, ws)
    torch.cuda.synchronize()
    want = O.segment_projection(kv, w["sigma_stale"], w["w_seg"], w["b_seg"], t.head_dim, "bf16")
    assert_close(to_host(y), want, 4e-3, 2.5e-2, f"segment projection {name}")
