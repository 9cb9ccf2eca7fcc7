"""The attention-mask ablations of App. F (A1 token-causal, A2 bidirectional,
A3 block-diagonal, next to the method's A0 block-causal mask) on the GPU,
through the C ABI, against the oracle."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import cr
from parity_util import as_f64, assert_close, to_dev, to_host
from test_gpu_parity import (GpuRun, _sample_rows, check_assembly, check_request, lib,  # noqa: F401
                             oracle_assemble, oracle_request)

pytestmark = pytest.mark.gpu

MODES = ["block_causal", "token_causal", "bidirectional", "block_diagonal"]

# request chunk lengths: one chunk; unit chunks; a ragged map over several tiles;
# several requests; a long first chunk whose end falls just past a query-tile
# start, so that the second query tile of a pair starts six key tiles later
# than the first under A3 and some rows see nothing of their first key tiles
MAPS = [[[300]], [[1] * 150], [[130, 77, 200, 1, 95]], [[129, 40], [5], [300, 256, 3]],
        [[800, 400]], [[100, 1000, 37], [256]]]


def _maps(reqs):
    """Request-local chunk end and start per token, chunk ids, cu_seqlens (from the lengths)."""
    cend, cstart, cids = [], [], []
    for r in reqs:
        e = np.cumsum(r)
        for i, n in enumerate(r):
            cend.append(np.full(n, e[i], np.int32))
            cstart.append(np.full(n, e[i] - n, np.int32))
        cids.append(np.concatenate([np.full(n, i, np.int32) for i, n in enumerate(r)]))
    cu = np.concatenate([[0], np.cumsum([sum(r) for r in reqs])]).astype(np.int32)
    return np.concatenate(cend), np.concatenate(cstart), cids, cu


@pytest.mark.parametrize("reqs", MAPS)
def test_chunk_starts_bit_exact(reqs):
    cend, cstart, _, cu = _maps(reqs)
    out = torch.full((len(cend),), -7, dtype=torch.int32, device="cuda")
    cr.cr_chunk_starts(to_dev(cend), cu, len(cend), out)
    torch.cuda.synchronize()
    assert np.array_equal(to_host(out), cstart)


@pytest.mark.parametrize("mode", MODES)
@pytest.mark.parametrize("reqs", MAPS)
@pytest.mark.parametrize("hd", [64, 32])
def test_masked_attention(hd, reqs, mode):
    g = np.random.default_rng(hd + sum(map(sum, reqs)) + MODES.index(mode))
    nh = 4 if hd == 32 else 8
    db = nh * hd
    cend, cstart, cids, cu = _maps(reqs)
    N = int(cu[-1])
    qkv = F.f32_to_bf16(g.standard_normal((N, 3 * db)).astype(np.float32))
    out = torch.full((N, db), float("nan"), dtype=torch.bfloat16, device="cuda")
    cs_dev = torch.empty(N, dtype=torch.int32, device="cuda")
    ce_dev = to_dev(cend)
    cr.cr_chunk_starts(ce_dev, cu, N, cs_dev)
    cr.cr_masked_attention(to_dev(qkv), db, nh, mode, ce_dev, cs_dev, cu, out)
    torch.cuda.synchronize()
    got = as_f64(to_host(out))
    q = as_f64(qkv)
    want, mag = np.empty((N, db)), np.empty((N, db))
    for r in range(len(reqs)):
        a, b = cu[r], cu[r + 1]
        sl = lambda off: q[a:b, off:off + db].reshape(b - a, nh, hd)
        m = O.attention_mask(cids[r], mode)
        want[a:b] = O.masked_attention(sl(0), sl(db), sl(2 * db), m).reshape(b - a, db)
        mag[a:b] = O.masked_attention(sl(0), sl(db), np.abs(sl(2 * db)), m).reshape(b - a, db)
    assert not np.isnan(got).any()
    # P is rounded to bf16 before the PV product and the output once to bf16 (as in
    # the block-causal test): |err| <= 2^-9 mag + 2^-9 |o|, with a 2x margin
    bound = 2.0 ** -8 * mag + 2.0 ** -8 * np.abs(want) + 1e-5
    worst = float((np.abs(got - want) / bound).max())
    assert worst <= 1.0, f"{mode} hd={hd} {reqs}: error / bound = {worst:.3f}"


@pytest.mark.parametrize("reqs", MAPS[2:4])
def test_block_causal_mode_is_the_chunk_causal_call(reqs):
    """A0 through the masked entry point is the method's attention, bit for bit."""
    g = np.random.default_rng(5)
    nh, hd = 8, 64
    db = nh * hd
    cend, _, _, cu = _maps(reqs)
    N = int(cu[-1])
    qkv = to_dev(F.f32_to_bf16(g.standard_normal((N, 3 * db)).astype(np.float32)))
    o1 = torch.empty(N, db, dtype=torch.bfloat16, device="cuda")
    o2 = torch.empty(N, db, dtype=torch.bfloat16, device="cuda")
    cr.cr_chunk_causal_attention(qkv, db, nh, to_dev(cend), cu, o1)
    cr.cr_masked_attention(qkv, db, nh, "block_causal", to_dev(cend), None, cu, o2)
    torch.cuda.synchronize()
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))


# ------------------------------------------------------------------ whole forward under each mask
@pytest.mark.parametrize("mode", MODES[1:])
@pytest.mark.parametrize("name", ["small", "small_multi"])
def test_forward_parity_masked(name, mode):
    case = F.make_case(name)
    g = GpuRun(case, mask_mode=mode)
    a = oracle_assemble(case)
    check_assembly(g, a)
    for r in range(len(a["cu_seqlens"]) - 1):
        res = oracle_request(case, a, r, mask_mode=mode)
        print(name, mode, r, check_request(case, g, a, r, res, tag=f"{name} mask={mode}"))


def test_block_diagonal_chunks_independent_on_gpu():
    """A3: perturbing one chunk leaves every output row of the other chunks bit-identical."""
    case = F.make_case("small")
    kvp, embp = case.pool()
    g1 = GpuRun(case, pool=(kvp, embp), mask_mode="block_diagonal")
    p = case.plan
    c = p.chunk_idx[2]                      # the request's third chunk
    kv2, emb2 = kvp.copy(), embp.copy()
    rng = np.random.default_rng(9)
    s0, n = p.chunk_start[c], p.chunk_len[c]
    kv2[s0:s0 + n] = F.f32_to_bf16(rng.standard_normal((n, kvp.shape[1])).astype(np.float32))
    emb2[s0:s0 + n] = F.f32_to_bf16(0.02 * rng.standard_normal((n, embp.shape[1])).astype(np.float32))
    g2 = GpuRun(case, pool=(kv2, emb2), mask_mode="block_diagonal")
    rows = g1.chunk_id == 2
    for x, y in ((g1.yf, g2.yf), (g1.kv, g2.kv)):
        assert np.array_equal(x[~rows], y[~rows])
        assert not np.array_equal(x[rows], y[rows])


@pytest.mark.slow
@pytest.mark.parametrize("mode", ["token_causal", "block_diagonal"])
def test_forward_parity_masked_full_size(mode):
    """The 8B-shape request (10 chunks of 512) under A1 and A3, sampled rows."""
    case = F.make_case("llama8b")
    g = GpuRun(case, mask_mode=mode)
    a = oracle_assemble(case)
    rows = _sample_rows(a["chunk_id"], 96)
    res = oracle_request(case, a, 0, rows=rows, mask_mode=mode)
    print(mode, check_request(case, g, a, 0, res, rows=rows, tag=f"{case.recipe.name} mask={mode}"))
