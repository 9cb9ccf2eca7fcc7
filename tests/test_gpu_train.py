"""One training update of the repair network (Sec. 4.2, App. A) on the GPU through
cr_train_step, against the oracle's training step."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from oracle import training as T
from paper_2609_35139_gb300 import TrainSession, cr, dims_from
from parity_util import to_dev
from test_gpu_parity import lib  # noqa: F401

pytestmark = pytest.mark.gpu


def _joint(case, kv_stale, seed=7):
    """A synthetic joint cache: the stale cache plus sigma_Delta-scaled noise, in cache dtype."""
    g = np.random.default_rng(seed)
    st = O.dtype_to_f64(kv_stale, case.target.cache_dtype)
    j = st + case.weights["sigma_delta"].astype(np.float64)[None] * g.standard_normal(st.shape)
    return O.round_to_cache(j, case.target.cache_dtype)


def _batch(case):
    kvp, embp = case.pool()
    p = case.plan
    a = O.assemble_stale(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    a["kv_joint"] = _joint(case, a["kv"])
    return a


def _session(case, a):
    t, r = dims_from(case.target, case.repairer)
    n = len(a["kv"])
    ts = TrainSession(t, r, case.weights, n, int(np.diff(a["cu_seqlens"]).max()))
    dev = dict(kv=to_dev(a["kv"]), kj=to_dev(a["kv_joint"]), emb=to_dev(a["emb"]),
               ce=to_dev(a["chunk_end"]), pos=to_dev(a["pos"]))
    return ts, dev, n


def _step(ts, dev, a, n, lr, mask="block_causal"):
    st = ts.step(dev["kv"], dev["kj"], dev["emb"], dev["ce"], dev["pos"], a["cu_seqlens"], n, lr,
                 mask_mode=mask)
    torch.cuda.synchronize()
    return st.cpu().numpy().copy()


def _tensor(ts, flat, name, shape):
    return ts.view(flat, name)[:int(np.prod(shape))].cpu().numpy().astype(np.float64).reshape(shape)


@pytest.mark.parametrize("name,mask", [("small", "block_causal"), ("small_multi", "block_causal"),
                                       ("small_multi", "token_causal"), ("small_multi", "bidirectional"),
                                       ("small_multi", "block_diagonal"), ("small_heads32", "block_causal")])
def test_train_step_matches_oracle(name, mask):
    if name == "small_heads32":   # 8 attention heads of 32 (the backward's other head size)
        case = F.make_case("small", repairer=F.RepairerDims(8, 128, 256, 2, 8, 1024))
    else:
        case = F.make_case(name)
    a = _batch(case)
    t, r = case.target, case.repairer
    names = T.trained_names(r.n_blocks)
    params = {k: (O.dtype_to_f64(case.weights[k], "bf16") if case.weights[k].dtype == np.uint16
                  else case.weights[k].astype(np.float64)) for k in names}
    zeros = {k: np.zeros_like(v) for k, v in params.items()}
    lr, hp = 1e-3, T.AdamWHyper()
    loss, norm, grads, _, _, _ = T.train_step(params, zeros, zeros, 1, lr, a,
                                              sigma_stale=case.weights["sigma_stale"],
                                              sigma_delta=case.weights["sigma_delta"], cache_dtype="bf16",
                                              head_dim=t.head_dim, n_heads=r.n_heads, hp=hp, mask_mode=mask)
    ts, dev, n = _session(case, a)
    stats = _step(ts, dev, a, n, lr, mask)
    g_loss, g_norm, g_coef = float(stats[0]), float(stats[1]), float(stats[2])
    print(name, mask, "loss", g_loss, loss, "norm", g_norm, norm)
    assert abs(g_loss - loss) <= 1e-3 * loss
    assert abs(g_norm - norm) <= 5e-3 * norm
    # The gradient, tensor by tensor.  The GPU rounds every GEMM operand (stored
    # activations, backward signals, weights) to bf16, 2^-9 relative, and
    # accumulates in fp32; the bound admits eight such roundings in RMS.
    g_gpu = {k: _tensor(ts, ts.grads, k, params[k].shape) for k in names}
    for k in names:
        gg, ref = g_gpu[k], grads[k]
        cos = float((gg * ref).sum() / np.sqrt((gg ** 2).sum() * (ref ** 2).sum()))
        rel = float(np.sqrt(np.mean((gg - ref) ** 2)) / np.sqrt(np.mean(ref ** 2)))
        print(f"  {k:14s} cos {cos:.6f} rel-RMS {rel:.3e}")
        assert cos >= 0.9999 and rel <= 1.5e-2, (k, cos, rel)
    # clipping and AdamW on the GPU's own gradient: the oracle's update, to fp32 rounding
    clipped, own_norm = T.clip_grads(g_gpu, hp.max_norm)
    assert abs(own_norm - g_norm) <= 1e-5 * own_norm
    assert abs(min(1.0, hp.max_norm / (own_norm + 1e-6)) - g_coef) <= 1e-6
    p1, m1, v1 = T.adamw_update(params, clipped, zeros, zeros, 1, lr, hp)
    for k in names:
        got = _tensor(ts, ts.params, k, params[k].shape)
        np.testing.assert_allclose(got, p1[k], rtol=2e-6, atol=1e-6 * lr, err_msg=k)
        np.testing.assert_allclose(_tensor(ts, ts.adam_m, k, params[k].shape), m1[k], rtol=1e-5,
                                   atol=1e-12, err_msg=k)
        np.testing.assert_allclose(_tensor(ts, ts.adam_v, k, params[k].shape), v1[k], rtol=1e-5,
                                   atol=1e-18, err_msg=k)
    # the bf16 copy is the rounding of the masters
    assert torch.equal(ts.params_bf16, ts.params.to(torch.bfloat16))


@pytest.mark.slow
def test_train_step_matches_oracle_8b_shapes():
    """The 8B shapes (D_KV 65536, d_b 1024, 6 blocks, 16 heads of 64) on a two-chunk
    request (1024 tokens): loss, norm and every gradient tensor against the oracle."""
    case = F.make_case("llama8b", n_req_chunks=2, requests=None)
    a = _batch(case)
    t, r = case.target, case.repairer
    names = T.trained_names(r.n_blocks)
    params = {k: (O.dtype_to_f64(case.weights[k], "bf16") if case.weights[k].dtype == np.uint16
                  else case.weights[k].astype(np.float64)) for k in names}
    zeros = {k: np.zeros_like(v) for k, v in params.items()}
    lr = 1e-4
    loss, norm, grads, _, _, _ = T.train_step(params, zeros, zeros, 1, lr, a,
                                              sigma_stale=case.weights["sigma_stale"],
                                              sigma_delta=case.weights["sigma_delta"], cache_dtype="bf16",
                                              head_dim=t.head_dim, n_heads=r.n_heads)
    ts, dev, n = _session(case, a)
    stats = _step(ts, dev, a, n, lr)
    print("8b shapes loss", stats[0], loss, "norm", stats[1], norm)
    assert abs(float(stats[0]) - loss) <= 1e-3 * loss
    assert abs(float(stats[1]) - norm) <= 5e-3 * norm
    for k in names:
        gg, ref = _tensor(ts, ts.grads, k, params[k].shape), grads[k]
        cos = float((gg * ref).sum() / np.sqrt((gg ** 2).sum() * (ref ** 2).sum()))
        rel = float(np.sqrt(np.mean((gg - ref) ** 2)) / np.sqrt(np.mean(ref ** 2)))
        print(f"  {k:14s} cos {cos:.6f} rel-RMS {rel:.3e}")
        assert cos >= 0.9999 and rel <= 1.5e-2, (k, cos, rel)


def test_train_steps_lower_the_loss():
    case = F.make_case("small_multi")
    a = _batch(case)
    ts, dev, n = _session(case, a)
    losses = [float(_step(ts, dev, a, n, 1e-3)[0]) for _ in range(4)]
    print(losses)
    assert losses[-1] < losses[0]
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, word
