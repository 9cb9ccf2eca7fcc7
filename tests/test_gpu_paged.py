"""cr_apply_residual_paged: the repaired rows written into a paged, layer-major
target cache match the oracle's repaired cache placed by the oracle's paged
scatter (App. A serving setup: loaded through the last complete 16-token block)
within the repaired-cache tolerance, and equal, bit for bit, the rows
cr_apply_residual repairs in place; tokens with a negative slot and unused slots
are left alone, the stale cache is not modified, and a slot out of range is
reported on the device and not written (the report makes the kernel's other
roles stop, as for any device-detected index error)."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import RepairSession, cr, dims_from, pack_host_weights
from parity_util import as_f64, half_ulp, to_dev, to_host

pytestmark = pytest.mark.gpu

SENTINEL = 0x7F7F   # a bf16 bit pattern the repair never produces here (about 3.4e38)


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


def _prepared(name="small"):
    case = F.make_case(name)
    t, r = dims_from(case.target, case.repairer)
    pw = pack_host_weights(case.weights, case.repairer.n_blocks)
    kvp, embp = case.pool()
    p = case.plan
    sess = RepairSession(t, r, pw, max_tokens=p.n_tokens)
    a = sess.assemble(to_dev(kvp), to_dev(embp), p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    sess.compress(a)
    sess.forward(a)
    return case, sess, a


@pytest.mark.parametrize("rope_mode", [cr.CR_ROPE_NONE, cr.CR_ROPE_GLOBAL])
def test_paged_write_equals_in_place_repair(rope_mode):
    case, sess, a = _prepared()
    n = a.n_tokens
    tg = case.target
    plane = tg.n_kv_heads * tg.head_dim
    planes = 2 * tg.n_layers
    stale = sess.kv[:n].clone()
    inv = case.inv_freq_target if rope_mode == cr.CR_ROPE_GLOBAL else None

    # blocks of 16 tokens in a shuffled order with spare blocks; the tail after
    # the last complete block is not written
    full = (n // 16) * 16
    n_blocks = n // 16 + 7
    order = np.random.default_rng(5).permutation(n_blocks)[: (n + 15) // 16]
    slots = np.full(n, -1, np.int64)
    tok = np.arange(full)
    slots[:full] = order[tok // 16] * 16 + tok % 16
    num_slots = n_blocks * 16
    paged = torch.full((planes, num_slots, plane), 0, dtype=torch.int16, device="cuda")
    paged.fill_(SENTINEL)
    paged = paged.view(torch.bfloat16)
    sess.apply_paged(a, to_dev(slots), paged, num_slots, inv, rope_mode)

    # reference: the in-place repair of a copy of the same stale rows
    ref = stale.clone()
    cr.cr_apply_residual(sess.target, sess.rep, sess.weights, sess.yf, n, ref, sess.pos, inv, rope_mode,
                         workspace=sess.workspace)
    torch.cuda.synchronize()
    assert torch.equal(sess.kv[:n], stale), "the stale cache must stay untouched"
    got = to_host(paged).reshape(planes, num_slots, plane)
    want = to_host(ref).reshape(n, planes, plane)
    written = np.zeros(num_slots, bool)
    written[slots[:full]] = True
    for pl in range(planes):
        assert np.array_equal(got[pl, slots[:full]], want[:full, pl]), f"plane {pl}"
        assert np.all(got[pl, ~written] == SENTINEL), f"plane {pl}: a slot not mapped was written"


def test_paged_slot_out_of_range_is_reported_and_skipped():
    case, sess, a = _prepared()
    n = a.n_tokens
    tg = case.target
    plane = tg.n_kv_heads * tg.head_dim
    num_slots = n
    slots = np.arange(n, dtype=np.int64)
    slots[3] = num_slots + 5
    paged = torch.empty((2 * tg.n_layers, num_slots, plane), dtype=torch.int16, device="cuda")
    paged.fill_(SENTINEL)
    sess.apply_paged(a, to_dev(slots), paged.view(torch.bfloat16), num_slots)
    st, word = cr.cr_get_device_status()
    cr.cr_clear_device_status()
    assert st == cr.CR_ERR_DEVICE_INDEX, word
    got = to_host(paged)
    assert np.all(got[:, 3] == SENTINEL)            # slot 3 belonged to the bad token only


@pytest.mark.parametrize("rope_mode", [cr.CR_ROPE_NONE, cr.CR_ROPE_GLOBAL])
def test_paged_write_matches_oracle(rope_mode):
    case, sess, a = _prepared()
    n = a.n_tokens
    tg = case.target
    L, H, dh = tg.n_layers, tg.n_kv_heads, tg.head_dim
    plane, planes = H * dh, 2 * L
    rope = rope_mode == cr.CR_ROPE_GLOBAL
    inv = case.inv_freq_target if rope else None
    # the request's blocks in a shuffled physical order among spare blocks
    n_phys = n // 16 + 9
    table = np.random.default_rng(11).permutation(n_phys)[: (n + 15) // 16]
    slots = O.paged_slot_mapping(n, table)
    num_slots = n_phys * 16
    paged = torch.empty((planes, num_slots, plane), dtype=torch.int16, device="cuda")
    paged.fill_(SENTINEL)
    sess.apply_paged(a, to_dev(slots), paged.view(torch.bfloat16), num_slots, inv, rope_mode)
    torch.cuda.synchronize()
    got = to_host(paged.view(torch.bfloat16)).reshape(planes, num_slots, plane)

    kvp, embp = case.pool()
    p = case.plan
    asm = O.assemble_stale(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    res = O.repair_request(asm["kv"], asm["emb"], asm["chunk_id"], asm["pos"], case.weights,
                           cache_dtype="bf16", n_layers=L, n_kv_heads=H, head_dim=dh,
                           n_heads=case.repairer.n_heads,
                           inv_freq_target=case.inv_freq_target if rope else None)
    exact = res.repaired_rot if rope else res.repaired
    want = O.paged_scatter(exact, slots, np.full((planes, num_slots, plane), np.nan), L, H, dh)
    written = ~np.isnan(want[:, :, 0])
    assert int(written[0].sum()) == (n // 16) * 16
    g64 = as_f64(got)
    worst = 0.0
    for pl in range(planes):
        w = written[pl]
        assert np.all(got[pl, ~w] == SENTINEL), f"plane {pl}: a slot outside the mapping was written"
        e, gg = want[pl, w], g64[pl, w]
        rms = np.sqrt(np.mean(e ** 2))
        err = float(np.maximum(np.abs(gg - e) - half_ulp(e, "bf16"), 0.0).max() / rms)
        cos = float((gg * e).sum() / np.sqrt((gg ** 2).sum() * (e ** 2).sum()))
        worst = max(worst, err)
        assert err <= 2e-2 and cos >= 0.999, f"plane {pl}: max err {err:.3e} x RMS, cosine {cos:.6f}"
    print(f"paged write vs oracle (rope={rope}): worst max err {worst:.3e} x RMS")


@pytest.mark.parametrize("name", ["small", "tiny"])
def test_target_rope_angles_from_table_equal_inline(name):
    """Under R_M the head reads each row's (cos, sin) from the per-call table written
    into the workspace; without a workspace it evaluates them in the epilogue.  Both
    evaluate the same formula (the angle's product error folded back in), compiled
    in different places, so they may differ in the last bit of an angle: the two
    repaired caches agree to one bf16 rounding (almost all values equal) or, for an
    fp32 cache, to 2^-20 of its RMS."""
    case, sess, a = _prepared(name)
    n = a.n_tokens
    stale = sess.kv[:n].clone()
    outs = []
    for ws in (sess.workspace, None):
        kv = stale.clone()
        cr.cr_apply_residual(sess.target, sess.rep, sess.weights, sess.yf, n, kv, sess.pos,
                             case.inv_freq_target, cr.CR_ROPE_GLOBAL, workspace=ws)
        torch.cuda.synchronize()
        outs.append(to_host(kv))
    dt = case.target.cache_dtype
    x, y = as_f64(outs[0]), as_f64(outs[1])
    if dt == "bf16":   # one rounding of the cache dtype
        bound = 2.0 * half_ulp(np.maximum(np.abs(x), np.abs(y)), dt)
    else:              # an angle's last bit moves a rotated pair by ~2^-23 of its size
        bound = 2.0 ** -20 * np.sqrt(np.mean(x ** 2))
    assert np.all(np.abs(x - y) <= bound), float(np.abs(x - y).max())
    if dt == "bf16":   # the coarse rounding absorbs almost every such difference
        assert np.mean(x != y) < 1e-2
