"""Output choices of App. F (correction applied to K only or V only, the zero
output offset of A5, each request's first chunk kept stale) and the stale
cache's re-rotation of K (Sec. 2.2) on the GPU, through the C ABI, against
the oracle."""
import itertools

import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import RepairSession, cr, dims_from, pack_host_weights
from parity_util import as_f64, check_repaired_cache, to_dev, to_host
from test_gpu_parity import _sample_rows, lib, oracle_assemble, oracle_request  # noqa: F401

pytestmark = pytest.mark.gpu


class Chain:
    """Assembly, features and blocks once; the stale cache is restored before each apply."""

    def __init__(self, case):
        t, r = dims_from(case.target, case.repairer)
        self.case, self.t = case, case.target
        self.pw = pack_host_weights(case.weights, case.repairer.n_blocks)
        kvp, embp = case.pool()
        p = case.plan
        self.s = RepairSession(t, r, self.pw, max_tokens=p.n_tokens)
        self.a = self.s.assemble(to_dev(kvp), to_dev(embp), p.chunk_start, p.chunk_len, p.chunk_idx,
                                 p.cu_chunks)
        self.s.compress(self.a)
        self.s.forward(self.a)
        self.n = n = self.a.n_tokens
        self.stale_dev = self.s.kv[:n].clone()
        torch.cuda.synchronize()
        self.stale = to_host(self.stale_dev)
        self.yf = to_host(self.s.yf[:n])
        self.pos = to_host(self.s.pos[:n])
        self.cid = to_host(self.s.chunk_id[:n])

    def apply(self, rope=False, **kw):
        self.s.kv[:self.n].copy_(self.stale_dev)
        self.s.apply(self.a, self.case.inv_freq_target,
                     cr.CR_ROPE_GLOBAL if rope else cr.CR_ROPE_NONE, **kw)
        torch.cuda.synchronize()
        return to_host(self.s.kv[:self.n])

    def z_from_gpu_yf(self, rows=None):
        """The head output on the GPU's own y_f (float64 product of the stored values)."""
        w = self.case.weights
        W = O.dtype_to_f64(w["w_out"], "bf16") if w["w_out"].dtype == np.uint16 else w["w_out"]
        y = as_f64(self.yf if rows is None else self.yf[rows])
        return y @ np.asarray(W, np.float64).T + np.asarray(w["b_out"], np.float64)

    def dims(self):
        return dict(n_layers=self.t.n_layers, n_kv_heads=self.t.n_kv_heads, head_dim=self.t.head_dim)


@pytest.fixture(scope="module", params=["small_multi", "tiny"])
def chain(request):
    return Chain(F.make_case(request.param))


CHOICES = list(itertools.product(["k", "v", "kv"], ["stale", "zero"], [False, True], [False, True]))


@pytest.mark.parametrize("component,offset,keep,rope", CHOICES)
def test_output_choice_head(chain, component, offset, keep, rope):
    c = chain
    dt = c.t.cache_dtype
    got = c.apply(rope=rope, component=component, offset=offset, keep_first_chunk=keep)
    keep_rows = (c.cid == 0) if keep else None
    exact = O.apply_output_choice(c.stale, c.z_from_gpu_yf(), c.case.weights["sigma_delta"],
                                  cache_dtype=dt, component=component, offset=offset,
                                  keep_rows=keep_rows, pos=c.pos,
                                  inv_freq_target=c.case.inv_freq_target if rope else None,
                                  **c.dims())
    check_repaired_cache(got, exact, c.t, dt)
    sel = O.component_columns(component, **c.dims())
    kcols = O.component_columns("k", **c.dims())
    # coordinates the choice leaves alone are the stale bits (V always; K too without R_M)
    untouched = ~sel & (~kcols if rope else np.ones_like(sel))
    bits = lambda x: np.ascontiguousarray(x).view(np.uint8 if dt == "bf16" else np.uint32)
    assert np.array_equal(bits(got[:, untouched]), bits(c.stale[:, untouched]))
    if keep:
        rows = c.cid == 0
        cols = ~kcols if rope else np.ones_like(sel)
        assert np.array_equal(bits(got[rows][:, cols]), bits(c.stale[rows][:, cols]))


def test_output_choice_whole_chain():
    """K only, first chunk kept, target R_M: the whole chain against the oracle's own head."""
    case = F.make_case("small_multi")
    c = Chain(case)
    got = c.apply(rope=True, component="k", keep_first_chunk=True)
    a = oracle_assemble(case)
    for r in range(len(a["cu_seqlens"]) - 1):
        lo, hi = a["cu_seqlens"][r], a["cu_seqlens"][r + 1]
        res = oracle_request(case, a, r)
        exact = O.apply_output_choice(a["kv"][lo:hi], res.z, case.weights["sigma_delta"],
                                      cache_dtype="bf16", component="k",
                                      keep_rows=a["chunk_id"][lo:hi] == 0, pos=a["pos"][lo:hi],
                                      inv_freq_target=case.inv_freq_target, **c.dims())
        print(r, check_repaired_cache(got[lo:hi], exact, case.target, "bf16"))


def test_rotate_k_is_the_stale_cache():
    case = F.make_case("small_multi")
    c = Chain(case)
    t = case.target
    s = c.s
    s.kv[:c.n].copy_(c.stale_dev)
    s.stale_kv(c.a, case.inv_freq_target)
    torch.cuda.synchronize()
    got = to_host(s.kv[:c.n])
    exact = O.stale_kv_cache_exact(c.stale, c.pos, case.inv_freq_target, cache_dtype="bf16",
                                   **c.dims())
    check_repaired_cache(got, exact, t, "bf16")
    vcols = O.component_columns("v", **c.dims())
    assert np.array_equal(got[:, vcols], c.stale[:, vcols])          # V as stored
    assert np.array_equal(got[c.pos == 0], c.stale[c.pos == 0])      # p = 0: identity
    # canonicalising the rotated cache gives the canonical cache back (two roundings)
    cr.cr_canonicalize_chunks(c.s.target, s.kv, c.n, s.pos, case.inv_freq_target)
    torch.cuda.synchronize()
    back = as_f64(to_host(s.kv[:c.n]))
    st = as_f64(c.stale)
    err = np.abs(back - st)[:, ~vcols]
    assert err.max() <= 2.0 ** -6 * np.abs(st[:, ~vcols]).max()
    assert np.sqrt(np.mean(err ** 2)) <= 2.0 ** -8 * np.sqrt(np.mean(st[:, ~vcols] ** 2))


@pytest.mark.slow
def test_output_choice_full_size_sampled():
    """The 8B-shape request: K only, zero offset, first chunk kept, target R_M; sampled rows."""
    case = F.make_case("llama8b")
    c = Chain(case)
    got = c.apply(rope=True, component="k", offset="zero", keep_first_chunk=True)
    rows = _sample_rows(c.cid, 96)
    exact = O.apply_output_choice(c.stale[rows], c.z_from_gpu_yf(rows), case.weights["sigma_delta"],
                                  cache_dtype="bf16", component="k", offset="zero",
                                  keep_rows=c.cid[rows] == 0, pos=c.pos[rows],
                                  inv_freq_target=case.inv_freq_target, **c.dims())
    print(check_repaired_cache(got[rows], exact, case.target, "bf16"))
    vcols = O.component_columns("v", **c.dims())
    assert np.array_equal(got[:, vcols], c.stale[:, vcols])
