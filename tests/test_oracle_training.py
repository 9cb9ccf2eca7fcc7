"""Pins for the training-step oracle (Sec. 4.2, App. A).

The backward is pinned by central finite differences of the loss on sampled
entries of every trained tensor and by torch autograd through an independent
float64 statement of the forward; the objective by closed forms; clipping and
AdamW by torch's own routines; the schedule by the numbers App. A prints.
"""
import math

import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from oracle import training as T

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _joint(case, kv_stale, seed=7):
    """A synthetic joint cache: the stale cache plus sigma_Delta-scaled noise, in cache dtype."""
    g = np.random.default_rng(seed)
    st = O.dtype_to_f64(kv_stale, case.target.cache_dtype)
    j = st + case.weights["sigma_delta"].astype(np.float64)[None] * g.standard_normal(st.shape)
    return O.round_to_cache(j, case.target.cache_dtype)


@pytest.fixture(scope="module")
def setup():
    case = F.make_case("tiny", requests=[[0, 1], [2]], n_req_chunks=None)
    kvp, embp = case.pool()
    p = case.plan
    a = O.assemble_stale(kvp, embp, p.chunk_start, p.chunk_len, p.chunk_idx, p.cu_chunks)
    a["kv_joint"] = _joint(case, a["kv"])
    names = T.trained_names(case.repairer.n_blocks)
    params = {k: case.weights[k].astype(np.float64) if case.weights[k].dtype != np.uint16
              else O.dtype_to_f64(case.weights[k], "bf16") for k in names}
    wf = T.forward_weights(params)
    wf["sigma_stale"] = case.weights["sigma_stale"]
    wf["sigma_delta"] = case.weights["sigma_delta"]
    return case, a, names, params, wf


def _loss(case, a, wf, mask="block_causal"):
    t, r = case.target, case.repairer
    c = T.train_forward(a["kv"], a["emb"], a["chunk_id"], a["pos"], a["cu_seqlens"], wf,
                        cache_dtype=t.cache_dtype, head_dim=t.head_dim, n_heads=r.n_heads, mask_mode=mask)
    loss, dz = T.train_loss(c.z, a["kv"], a["kv_joint"], wf["sigma_delta"], a["cu_seqlens"],
                            t.cache_dtype)
    return loss, dz, c


def _grads(case, a, wf, mask="block_causal"):
    t, r = case.target, case.repairer
    loss, dz, c = _loss(case, a, wf, mask)
    g = T.train_backward(c, dz, wf, a["pos"], a["cu_seqlens"], O.dtype_to_f64(a["emb"], t.cache_dtype),
                         head_dim=t.head_dim, n_heads=r.n_heads)
    return loss, g


def test_forward_matches_inference_oracle(setup):
    """The training forward's y_f and repaired cache equal the inference oracle's (per request)."""
    case, a, names, params, wf = setup
    t, r = case.target, case.repairer
    _, _, c = _loss(case, a, wf)
    w = dict(case.weights)
    for k in names:
        w[k] = wf[k]
    for q in range(len(a["cu_seqlens"]) - 1):
        lo, hi = a["cu_seqlens"][q], a["cu_seqlens"][q + 1]
        res = O.repair_request(a["kv"][lo:hi], a["emb"][lo:hi], a["chunk_id"][lo:hi], a["pos"][lo:hi], w,
                               cache_dtype=t.cache_dtype, n_layers=t.n_layers, n_kv_heads=t.n_kv_heads,
                               head_dim=t.head_dim, n_heads=r.n_heads)
        np.testing.assert_allclose(c.yf[lo:hi], res.yf, rtol=1e-10, atol=1e-10)
        np.testing.assert_allclose(c.z[lo:hi], res.z, rtol=1e-9, atol=1e-10)


def test_backward_matches_finite_differences(setup):
    case, a, names, params, wf = setup
    _, g = _grads(case, a, wf)
    assert set(g) == set(names)
    rng = np.random.default_rng(11)
    for k in names:
        flat = wf[k].reshape(-1)
        for idx in rng.choice(flat.size, size=min(3, flat.size), replace=False):
            h = 1e-4 * max(1.0, abs(flat[idx]))
            w2 = dict(wf)
            w2[k] = wf[k].copy()
            w2[k].reshape(-1)[idx] += h
            lp = _loss(case, a, w2)[0]
            w2[k].reshape(-1)[idx] -= 2 * h
            lm = _loss(case, a, w2)[0]
            fd = (lp - lm) / (2 * h)
            an = g[k].reshape(-1)[idx]
            assert abs(fd - an) <= 1e-6 * max(1e-3, abs(fd)) + 1e-9, (k, idx, fd, an)


def _torch_loss(case, a, wt, mask="block_causal"):
    """The same objective stated with torch ops (float64), for autograd."""
    t, r = case.target, case.repairer
    n = a["kv"].shape[0]
    kv = torch.from_numpy(O.dtype_to_f64(a["kv"], t.cache_dtype))
    emb = torch.from_numpy(O.dtype_to_f64(a["emb"], t.cache_dtype))
    x = kv / torch.from_numpy(case.weights["sigma_stale"].astype(np.float64))
    S = x.shape[1] // t.head_dim
    y = torch.einsum("tsj,sij->tsi", x.reshape(n, S, t.head_dim), wt["w_seg"]) + wt["b_seg"]
    y = y.reshape(n, -1)
    s = y @ wt["w_map"].T + wt["b_map"]
    e = emb @ wt["w_tok"].T + wt["b_tok"]
    h = torch.cat([s, e], 1) @ wt["w_fuse"].T + wt["b_fuse"]
    db, nh = h.shape[1], r.n_heads
    d = db // nh
    pos = torch.from_numpy(a["pos"].astype(np.float64))
    ang = pos[:, None] * torch.from_numpy(O.repair_inv_freq(d, 1e4))[None]
    cos, sin = torch.cos(ang)[:, None], torch.sin(ang)[:, None]

    def rope(u):
        p, q = u[..., :d // 2], u[..., d // 2:]
        return torch.cat([p * cos - q * sin, q * cos + p * sin], -1)

    ln = lambda u, gname, bname: torch.nn.functional.layer_norm(u, (db,), wt[gname], wt[bname], 1e-5)
    for b in range(case.repairer.n_blocks):
        pre = f"blk{b}."
        xin = h + s @ wt["w_rein"][b].T + wt["b_rein"][b]
        qkv = ln(xin, pre + "ln1_g", pre + "ln1_b") @ wt[pre + "w_qkv"].T + wt[pre + "b_qkv"]
        q = rope(qkv[:, :db].reshape(n, nh, d))
        k = rope(qkv[:, db:2 * db].reshape(n, nh, d))
        v = qkv[:, 2 * db:].reshape(n, nh, d)
        outs = []
        for rq in range(len(a["cu_seqlens"]) - 1):
            lo, hi = a["cu_seqlens"][rq], a["cu_seqlens"][rq + 1]
            m = torch.from_numpy(O.attention_mask(a["chunk_id"][lo:hi], mask))
            o = torch.nn.functional.scaled_dot_product_attention(
                q[lo:hi].transpose(0, 1), k[lo:hi].transpose(0, 1), v[lo:hi].transpose(0, 1), attn_mask=m)
            outs.append(o.transpose(0, 1))
        att = torch.cat(outs).reshape(n, db)
        xm = xin + att @ wt[pre + "w_o"].T + wt[pre + "b_o"]
        gl = torch.nn.functional.gelu(ln(xm, pre + "ln2_g", pre + "ln2_b") @ wt[pre + "w_fc1"].T
                                      + wt[pre + "b_fc1"])
        h = xm + gl @ wt[pre + "w_fc2"].T + wt[pre + "b_fc2"]
    z = ln(h, "lnf_g", "lnf_b") @ wt["w_out"].T + wt["b_out"]
    tgt = (torch.from_numpy(O.dtype_to_f64(a["kv_joint"], t.cache_dtype)) - kv) \
        / torch.from_numpy(case.weights["sigma_delta"].astype(np.float64))
    total = 0.0
    nreq = len(a["cu_seqlens"]) - 1
    for rq in range(nreq):
        lo, hi = a["cu_seqlens"][rq], a["cu_seqlens"][rq + 1]
        total = total + ((z[lo:hi] - tgt[lo:hi]) ** 2).mean() / nreq
    return total


@pytest.mark.parametrize("mask", O.MASK_MODES)
def test_backward_matches_torch_autograd(setup, mask):
    """Every attention mask (the method's and the App. F ablations) through the same backward."""
    case, a, names, params, wf = setup
    loss, g = _grads(case, a, wf, mask)
    wt = {k: torch.tensor(wf[k], dtype=torch.float64, requires_grad=True) for k in names}
    tl = _torch_loss(case, a, wt, mask)
    tl.backward()
    assert abs(float(tl.detach()) - loss) <= 1e-12 * abs(loss)
    for k in names:
        ref = wt[k].grad.numpy()
        np.testing.assert_allclose(g[k], ref, rtol=1e-8, atol=1e-12 * np.abs(ref).max() + 1e-300,
                                   err_msg=k)


def test_loss_closed_forms(setup):
    case, a, _, _, wf = setup
    t = case.target
    sd = case.weights["sigma_delta"]
    tgt = (O.dtype_to_f64(a["kv_joint"], t.cache_dtype) - O.dtype_to_f64(a["kv"], t.cache_dtype)) \
        / sd.astype(np.float64)[None]
    loss, dz = T.train_loss(tgt.copy(), a["kv"], a["kv_joint"], sd, a["cu_seqlens"], t.cache_dtype)
    assert loss == 0.0 and not dz.any()
    # z = target + 1 everywhere: every request's mean square is 1
    loss, dz = T.train_loss(tgt + 1.0, a["kv"], a["kv_joint"], sd, a["cu_seqlens"], t.cache_dtype)
    assert abs(loss - 1.0) < 1e-12
    n0 = a["cu_seqlens"][1]
    np.testing.assert_allclose(dz[:n0], 2.0 / (n0 * tgt.shape[1]) / 2, rtol=1e-12)


def test_clip_matches_torch():
    g = np.random.default_rng(3)
    grads = {"a": g.standard_normal((5, 7)), "b": g.standard_normal(11) * 3}
    for scale in (0.01, 10.0):
        gs = {k: v * scale for k, v in grads.items()}
        clipped, norm = T.clip_grads(gs, 1.0)
        ts = [torch.tensor(v, requires_grad=True) for v in gs.values()]
        for tt, v in zip(ts, gs.values()):
            tt.grad = torch.tensor(v)
        tn = torch.nn.utils.clip_grad_norm_(ts, 1.0)
        assert abs(float(tn) - norm) <= 1e-12 * norm
        for tt, k in zip(ts, gs):
            np.testing.assert_allclose(clipped[k], tt.grad.numpy(), rtol=1e-12)


def test_adamw_matches_torch():
    g = np.random.default_rng(4)
    hp = T.AdamWHyper()
    p = {"w": g.standard_normal((4, 3)), "b": g.standard_normal(5)}
    tp = [torch.tensor(v, requires_grad=True) for v in p.values()]
    opt = torch.optim.AdamW(tp, lr=3e-4, betas=(hp.beta1, hp.beta2), eps=hp.eps,
                            weight_decay=hp.weight_decay)
    m = {k: np.zeros_like(v) for k, v in p.items()}
    v = {k: np.zeros_like(x) for k, x in p.items()}
    for step in range(1, 4):
        lr = 1e-4 * step
        for group in opt.param_groups:
            group["lr"] = lr
        grads = {k: g.standard_normal(x.shape) for k, x in p.items()}
        for tt, k in zip(tp, p):
            tt.grad = torch.tensor(grads[k])
        opt.step()
        p, m, v = T.adamw_update(p, grads, m, v, step, lr, hp)
        for tt, k in zip(tp, p):
            np.testing.assert_allclose(p[k], tt.detach().numpy(), rtol=1e-12, atol=1e-15)


def test_lr_schedule_matches_paper():
    """App. A: 2,000 warmup updates to 3e-4, cosine decay toward 3e-5 over 100,000 updates;
    the controlled comparisons: 500 warmup updates over 25,000."""
    assert T.lr_schedule(2000) == pytest.approx(3e-4, rel=1e-12)
    assert T.lr_schedule(1000) == pytest.approx(1.5e-4, rel=1e-12)
    assert T.lr_schedule(100000) == pytest.approx(3e-5, rel=1e-12)
    assert T.lr_schedule(51000) == pytest.approx(1.65e-4, rel=1e-12)    # cosine midpoint
    lrs = [T.lr_schedule(s) for s in range(2000, 100001, 997)]
    assert all(x >= y for x, y in zip(lrs, lrs[1:]))
    assert T.lr_schedule(500, warmup=500, total=25000) == pytest.approx(3e-4, rel=1e-12)
    assert T.lr_schedule(25000, warmup=500, total=25000) == pytest.approx(3e-5, rel=1e-12)


def test_train_step_reduces_loss(setup):
    """A few updates at a fixed rate lower the objective (the whole step is consistent)."""
    case, a, names, params, _ = setup
    t, r = case.target, case.repairer
    m = {k: np.zeros_like(v) for k, v in params.items()}
    v = {k: np.zeros_like(x) for k, x in params.items()}
    p = params
    losses = []
    for step in range(1, 5):
        loss, norm, _, p, m, v = T.train_step(p, m, v, step, 1e-3, a, sigma_stale=case.weights["sigma_stale"],
                                              sigma_delta=case.weights["sigma_delta"],
                                              cache_dtype=t.cache_dtype, head_dim=t.head_dim,
                                              n_heads=r.n_heads)
        losses.append(loss)
    assert losses[-1] < losses[0]
