"""RepairPipeline (host transfers overlapped with repair on two slots) returns
exactly what a plain RepairSession returns for each request, through several
reuses of each slot, and each request's repaired cache, read back into host
memory, matches the oracle's within the repaired-cache tolerance."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import RepairPipeline, RepairSession, cr, dims_from, pack_host_weights
from parity_util import check_repaired_cache, to_dev, to_host

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


def _pinned(a):
    a = np.ascontiguousarray(a)
    t = torch.from_numpy(a.view(np.int16)).view(torch.bfloat16) if a.dtype == np.uint16 else torch.from_numpy(a)
    return t.pin_memory()


def test_pipeline_matches_session_per_request():
    case = F.make_case("small_multi")
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    reqs = [p.chunk_idx[p.cu_chunks[i]:p.cu_chunks[i + 1]] for i in range(len(p.cu_chunks) - 1)]
    assert len(reqs) >= 2
    lens = [int(p.chunk_len[s].sum()) for s in reqs]
    cap = max(lens)

    # reference: each request alone through a session, pool on the device
    sess = RepairSession(t, r, pw, max_tokens=cap)
    kvd, embd = to_dev(kvp), to_dev(embp)
    ref = []
    for sel in reqs:
        a = sess.repair(kvd, embd, p.chunk_start, p.chunk_len, sel.astype(np.int32),
                        np.array([0, len(sel)], np.int32))
        torch.cuda.synchronize()
        ref.append(to_host(sess.kv[:a.n_tokens]).copy())

    # pipeline: pinned host pool in, pinned host caches out; every slot used twice or more
    pipe = RepairPipeline(t, r, pw, max_tokens=cap)
    kv_h, emb_h = _pinned(kvp), _pinned(embp)
    order = [i % len(reqs) for i in range(max(5, 2 * len(reqs) + 1))]
    outs = [torch.empty(cap, sess.d_kv, dtype=kv_h.dtype).pin_memory() for _ in order]
    for k, i in enumerate(order):
        sel = reqs[i]
        pipe.submit(kv_h, emb_h, p.chunk_start[sel], p.chunk_len[sel], outs[k])
    pipe.drain()
    torch.cuda.synchronize()
    for k, i in enumerate(order):
        got = outs[k][:lens[i]].view(torch.int16).numpy().view(np.uint16) \
            if kv_h.dtype == torch.bfloat16 else outs[k][:lens[i]].numpy()
        assert np.array_equal(got.view(np.uint8), ref[i].view(np.uint8)), f"request {i} (submission {k})"
    # every request's host copy against the oracle (first submission of each)
    tg = case.target
    for i, sel in enumerate(reqs):
        k = order.index(i)
        got = outs[k][:lens[i]].view(torch.int16).numpy().view(np.uint16)
        kv_r = np.concatenate([kvp[p.chunk_start[c]:p.chunk_start[c] + p.chunk_len[c]] for c in sel])
        emb_r = np.concatenate([embp[p.chunk_start[c]:p.chunk_start[c] + p.chunk_len[c]] for c in sel])
        cid = np.concatenate([np.full(p.chunk_len[c], j, np.int32) for j, c in enumerate(sel)])
        res = O.repair_request(kv_r, emb_r, cid, np.arange(lens[i], dtype=np.int32), case.weights,
                               cache_dtype="bf16", n_layers=tg.n_layers, n_kv_heads=tg.n_kv_heads,
                               head_dim=tg.head_dim, n_heads=case.repairer.n_heads)
        check_repaired_cache(got, res.repaired, tg, "bf16", stale=kv_r)


def test_pipeline_rejects_oversize_request():
    case = F.make_case("small_multi")
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    pipe = RepairPipeline(t, r, pw, max_tokens=8)
    out = torch.empty(8, 1, dtype=torch.bfloat16).pin_memory()
    with pytest.raises(ValueError):
        pipe.submit(_pinned(kvp), _pinned(embp), p.chunk_start[:1], p.chunk_len[:1], out)
