"""The head that reads the stale rows from the chunk pool (cr_apply_residual_pool,
after cr_assemble_compress without an assembled cache) writes exactly the cache
that the in-place path writes (cr_assemble_compress into kv, the blocks, then
cr_apply_residual on kv), bit for bit: on chunk maps whose 128-row boxes are whole
pool ranges (10 x 512), on ragged maps whose boxes straddle chunks and the end of
the request, with several requests in one call, and under the target's R_M."""
import numpy as np
import pytest
import torch

import fixtures as F
from paper_2609_35139_gb300 import RepairSession, cr, dims_from, pack_host_weights
from parity_util import to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_35139_gb300 import build
    build.build()
    cr.lib()
    cr.cr_clear_device_status()
    yield
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, f"device status {word}"


def _both(case_name, rope):
    case = F.make_case(case_name)
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    kvd, embd = to_dev(kvp), to_dev(embp)
    freq = case.inv_freq_target if rope else None
    mode = cr.CR_ROPE_GLOBAL if rope else cr.CR_ROPE_NONE
    sess = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    # in place: the assembled cache, then the head on it
    a = sess.assemble_compress(kvd, embd, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    sess.forward(a)
    sess.apply(a, freq, mode)
    torch.cuda.synchronize()
    ref = to_host(sess.kv[:a.n_tokens]).copy()
    # from the pool: kv is cleared first, so every row must come from the head
    sess.kv.zero_()
    b = sess.assemble_compress(kvd, embd, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks,
                               write_kv=False)
    sess.forward(b)
    sess.apply_pool(b, kvd, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks, freq, mode)
    torch.cuda.synchronize()
    got = to_host(sess.kv[:b.n_tokens]).copy()
    return p, ref, got


@pytest.mark.parametrize("case_name,rope", [("llama8b", False), ("llama8b", True), ("qwen7b", False),
                                            ("small_multi", False), ("small", True)])
def test_pool_head_matches_in_place(case_name, rope):
    p, ref, got = _both(case_name, rope)
    assert ref.shape == got.shape
    ragged = bool(np.any(np.asarray(p.chunk_len)[np.asarray(p.chunk_idx)] % 128 != 0))
    diff = np.nonzero(ref.view(np.uint16) != got.view(np.uint16))
    assert diff[0].size == 0, (f"{case_name}: {diff[0].size} values differ (ragged map: {ragged}), "
                               f"first rows {np.unique(diff[0])[:8]}")


def test_repair_uses_the_pool_head():
    # RepairSession.repair under the method's output: the same cache as the
    # in-place composition (the parity tests compare repair() with the oracle)
    case = F.make_case("small")
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    kvd, embd = to_dev(kvp), to_dev(embp)
    sess = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    a = sess.repair(kvd, embd, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    torch.cuda.synchronize()
    got = to_host(sess.kv[:a.n_tokens]).copy()
    sess.kv.zero_()
    b = sess.assemble_compress(kvd, embd, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    sess.forward(b)
    sess.apply(b)
    torch.cuda.synchronize()
    ref = to_host(sess.kv[:b.n_tokens]).copy()
    assert np.array_equal(ref.view(np.uint16), got.view(np.uint16))


def test_pool_head_rejects_bad_plans():
    case = F.make_case("small")
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    kvd = to_dev(kvp)
    sess = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    # a chunk map of a different length than n_tokens
    with pytest.raises(cr.CrError):
        cr.cr_apply_residual_pool(t, r, pw, sess.yf, p.n_tokens - 1, kvd, p.chunk_start, p.chunk_len,
                                  p.chunk_idx, p.cu_chunks, sess.kv, sess.pos, workspace=sess.workspace)
    # a chunk index past the pool's chunks
    bad = np.array(p.chunk_idx, np.int32).copy()
    bad[0] = len(p.chunk_len)
    with pytest.raises(cr.CrError):
        cr.cr_apply_residual_pool(t, r, pw, sess.yf, p.n_tokens, kvd, p.chunk_start, p.chunk_len, bad,
                                  p.cu_chunks, sess.kv, sess.pos, workspace=sess.workspace)
    torch.cuda.synchronize()
