"""cr_assemble_compress (stale-cache assembly fused into the segment projection,
Sec. 4.1) against the two calls it replaces, and the fused repair chain against
the oracle.

The fused call must give every output of cr_assemble_stale + cr_compress_features
bit for bit: the assembled cache (written by the projection kernel's tile
stores), embeddings, chunk map, h^0 and the reinjection terms.  Chunk layouts
cover 128-row tiles with ragged tails, a 1-token chunk, a chunk that ends the
pool (its last tile reads past the pool, zero fill), up to 256 requests, 64- and
128-dim target heads, d_seg 8 and 16, and the fp32 cache (two-call path).
"""
from dataclasses import replace

import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import RepairSession, cr, dims_from, pack_host_weights
from parity_util import check_repaired_cache, residual_cosine, to_dev, to_host
from test_gpu_parity import lib  # noqa: F401

pytestmark = pytest.mark.gpu


def _case(name):
    if name == "small_dh64":   # 64-dim target heads, d_seg 16
        base = F.RECIPES["small"]
        rc = replace(base, name="small_dh64", target=F.TargetDims(4, 2, 64, 512, "bf16", 1e6),
                     repairer=F.RepairerDims(16, 128, 256, 2, 4, 1024))
        return F.make_case(rc)
    if name == "small_tail":   # the request ends with the pool's last (33-token) chunk
        return F.make_case("small_multi", requests=[[7], [4, 7, 3]])
    if name == "small_256req":   # the most requests one call takes
        return F.make_case("small_multi", requests=[[i % 8, (3 * i + 1) % 8] for i in range(256)])
    return F.make_case(name)


def _outputs(s, n, n_req):
    return dict(kv=s.kv[:n].clone(), emb=s.emb[:n].clone(), chunk_id=s.chunk_id[:n].clone(),
                chunk_end=s.chunk_end[:n].clone(), pos=s.pos[:n].clone(),
                cu=s.cu_seqlens[:n_req + 1].clone(), h0=s.h0[:n].clone(), rein=s.rein[:n].clone())


@pytest.mark.parametrize("name", ["small", "small_multi", "small_tail", "small_dh64", "small_256req",
                                  "tiny", "qwen3b", "qwen7b", "llama8b"])
def test_fused_matches_two_calls(name):
    case = _case(name)
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = (to_dev(x) for x in case.pool())
    p = case.plan
    n_req = len(p.cu_chunks) - 1
    s2 = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    a2 = s2.assemble(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    s2.compress(a2)
    ref = _outputs(s2, a2.n_tokens, n_req)
    del s2
    s1 = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    # poison the outputs: every row must be written by the fused call
    s1.kv.fill_(float("nan"))
    s1.h0.fill_(float("nan"))
    a1 = s1.assemble_compress(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    torch.cuda.synchronize()
    assert a1.n_tokens == a2.n_tokens == p.n_tokens
    assert np.array_equal(a1.cu_seqlens, a2.cu_seqlens)
    got = _outputs(s1, a1.n_tokens, n_req)
    for k in ref:
        a, b = got[k], ref[k]
        if a.dtype in (torch.bfloat16, torch.float32):
            a, b = a.view(torch.int16 if a.dtype == torch.bfloat16 else torch.int32), \
                b.view(torch.int16 if b.dtype == torch.bfloat16 else torch.int32)
        assert torch.equal(a, b), k
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, word


@pytest.mark.parametrize("name", ["small", "small_tail"])
def test_fused_repair_matches_oracle(name):
    """RepairSession.repair (the fused front, blocks, head) against the oracle on every
    repaired value of every request."""
    case = _case(name)
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp_h, embp_h = case.pool()
    p = case.plan
    s = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    a = s.repair(to_dev(kvp_h), to_dev(embp_h), p.chunk_start, p.chunk_len, p.chunk_idx,
                 p.cu_chunks)
    torch.cuda.synchronize()
    kv = to_host(s.kv[:a.n_tokens])
    asm = O.assemble_stale(kvp_h, embp_h, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    tgt, rp = case.target, case.repairer
    for q in range(len(p.cu_chunks) - 1):
        lo, hi = asm["cu_seqlens"][q], asm["cu_seqlens"][q + 1]
        res = O.repair_request(asm["kv"][lo:hi], asm["emb"][lo:hi], asm["chunk_id"][lo:hi],
                               asm["pos"][lo:hi], case.weights, cache_dtype=tgt.cache_dtype,
                               n_layers=tgt.n_layers, n_kv_heads=tgt.n_kv_heads,
                               head_dim=tgt.head_dim, n_heads=rp.n_heads)
        check_repaired_cache(kv[lo:hi], res.repaired, tgt, tgt.cache_dtype)
        cos = residual_cosine(kv[lo:hi], asm["kv"][lo:hi], res.repaired, tgt.cache_dtype)
        assert cos >= 0.99, (q, cos)
