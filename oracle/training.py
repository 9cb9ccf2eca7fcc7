"""Oracle for one training step of the repair network, in float64.

TEST INFRASTRUCTURE, like the rest of this package: imported only by the
tests and the benchmark's CPU legs; the product path never imports it.

  Sec. 4.2  "Paired cache supervision": the target residual is
            Delta KV^c* = KV^c_joint - KV^c_stale (both canonical).
            "Normalization and objective": for an example of N document
            tokens, L = 1/(N D_KV) sum_t || z_t - Delta KV^c*_t / sigma_Delta ||^2;
            every part of the network is trained (StaleEncoder, token
            projection, fusion, Repair Blocks, reinjection, output head);
            sigma_stale and sigma_Delta are fixed statistics.
  App. A    "Optimization": AdamW, (beta1, beta2) = (0.9, 0.95), weight decay
            0.01, unit gradient clipping, warmup then cosine learning rate.
  App. F    training keeps the repair weights in FP32.

The forward is the inference forward of oracle/cacherepair.py (Sec. 4.1)
with every intermediate kept; the backward is the chain rule through it,
written out by hand step by step in reverse order.  Matrices enter the
forward as the bf16 rounding of their fp32 masters (the GPU's mixed
precision); the gradient is taken with respect to those values.

Readings:
  R21 A batch of several requests is trained on the mean of the per-request
      losses (each normalised by its own N D_KV).
  R22 Unit gradient clipping is clipping of the global L2 norm over all
      trained parameters at 1: g <- g * min(1, 1 / (||g|| + 1e-6)).
  R23 AdamW is decoupled weight decay on every trained parameter (biases and
      LayerNorm parameters included): theta <- theta (1 - lr wd), then the
      bias-corrected Adam step lr m_hat / (sqrt(v_hat) + eps), eps = 1e-8.
  R24 Learning rate at update t (1-based): linear warmup from 0 to the peak
      over the warmup updates, then cosine decay from the peak to the final
      rate at the last update.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np
import torch

from .cacherepair import (attention_mask, dtype_to_f64, gelu, layer_norm, repair_inv_freq,
                          rope_rotate_half, round_to_cache)

__all__ = ["TRAINED", "MATRICES", "trained_names", "forward_weights", "train_forward",
           "train_loss", "train_backward", "grad_global_norm", "clip_grads", "adamw_update",
           "lr_schedule", "train_step", "TrainCache", "AdamWHyper"]

# trained tensors of the fixture's weight dict, in the fixture's order; the
# block tensors repeat per block
TOP_BEFORE = ["w_seg", "b_seg", "w_map", "b_map", "w_tok", "b_tok", "w_fuse", "b_fuse",
              "w_rein", "b_rein"]
BLOCK = ["ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ln2_g", "ln2_b", "w_fc1", "b_fc1",
         "w_fc2", "b_fc2"]
TOP_AFTER = ["lnf_g", "lnf_b", "w_out", "b_out"]
MATRICES = {"w_seg", "w_map", "w_tok", "w_fuse", "w_rein", "w_qkv", "w_o", "w_fc1", "w_fc2", "w_out"}
TRAINED = TOP_BEFORE + BLOCK + TOP_AFTER


def trained_names(n_blocks: int) -> List[str]:
    """Every trained tensor's key, in the order of the flat parameter vector."""
    return TOP_BEFORE + [f"blk{b}.{k}" for b in range(n_blocks) for k in BLOCK] + TOP_AFTER


def _is_matrix(name: str) -> bool:
    return name.split(".")[-1] in MATRICES


def _bf16_value(x: np.ndarray) -> np.ndarray:
    return dtype_to_f64(round_to_cache(np.asarray(x, np.float64), "bf16"), "bf16")


def forward_weights(params: Dict[str, np.ndarray]) -> Dict[str, np.ndarray]:
    """The values the forward uses: matrices rounded to bf16, vectors as they are."""
    return {k: (_bf16_value(v) if _is_matrix(k) else np.asarray(v, np.float64))
            for k, v in params.items()}


# ------------------------------------------------------------------ forward with every intermediate
@dataclass
class BlockCache:
    x_in: np.ndarray      # block input h^{b-1} + P_b(s)
    u1: np.ndarray        # LN1(x_in)
    q: np.ndarray         # after the repairer RoPE, [n, heads, d]
    k: np.ndarray
    v: np.ndarray
    P: List[np.ndarray]   # per request: softmax weights [heads, n_r, n_r]
    a: np.ndarray         # attention output [n, d_b]
    x_mid: np.ndarray     # x_in + O(a)
    u2: np.ndarray        # LN2(x_mid)
    pre: np.ndarray       # FC1(u2), before GELU
    g: np.ndarray         # GELU(pre)


@dataclass
class TrainCache:
    x: np.ndarray          # kv / sigma_stale, [n, D_KV]
    y: np.ndarray          # segment projections [n, S d_seg]
    s: np.ndarray          # StaleEncoder output [n, d_c]
    e: np.ndarray          # token projection [n, d_c]
    h0: np.ndarray
    blocks: List[BlockCache] = field(default_factory=list)
    hB: np.ndarray = None
    yf: np.ndarray = None
    z: np.ndarray = None


def train_forward(kv: np.ndarray, emb: np.ndarray, chunk_id: np.ndarray, pos: np.ndarray,
                  cu_seqlens: np.ndarray, wf: Dict[str, np.ndarray], *, cache_dtype: str,
                  head_dim: int, n_heads: int, eps: float = 1e-5, rope_theta: float = 1e4,
                  mask_mode: str = "block_causal") -> TrainCache:
    """The repair forward of Sec. 4.1 over a batch of requests (cu_seqlens), keeping
    what the backward needs.  wf: forward_weights(params) plus the fixed sigmas."""
    n = kv.shape[0]
    x = dtype_to_f64(kv, cache_dtype) / np.asarray(wf["sigma_stale"], np.float64)[None, :]
    S = x.shape[1] // head_dim
    W = wf["w_seg"]                                   # [S, d_seg, d_h]
    xs = x.reshape(n, S, head_dim)
    y = (np.einsum("tsj,sij->tsi", xs, W) + wf["b_seg"][None]).reshape(n, -1)
    s = y @ wf["w_map"].T + wf["b_map"]
    e = dtype_to_f64(emb, cache_dtype) @ wf["w_tok"].T + wf["b_tok"]
    h0 = np.concatenate([s, e], axis=1) @ wf["w_fuse"].T + wf["b_fuse"]
    c = TrainCache(x=x, y=y, s=s, e=e, h0=h0)
    h = h0
    B = wf["w_rein"].shape[0]
    db = h0.shape[1]
    dh = db // n_heads
    f = repair_inv_freq(dh, rope_theta)
    for b in range(B):
        p = {k: wf[f"blk{b}.{k}"] for k in BLOCK}
        x_in = h + (s @ wf["w_rein"][b].T + wf["b_rein"][b])
        u1 = layer_norm(x_in, p["ln1_g"], p["ln1_b"], eps)
        qkv = u1 @ p["w_qkv"].T + p["b_qkv"]
        q = rope_rotate_half(qkv[:, :db].reshape(n, n_heads, dh), pos, f)
        k = rope_rotate_half(qkv[:, db:2 * db].reshape(n, n_heads, dh), pos, f)
        v = qkv[:, 2 * db:].reshape(n, n_heads, dh)
        a = np.empty((n, n_heads, dh))
        Ps = []
        for r in range(len(cu_seqlens) - 1):
            lo, hi = int(cu_seqlens[r]), int(cu_seqlens[r + 1])
            mask = attention_mask(chunk_id[lo:hi], mask_mode)
            sc = np.einsum("ihd,jhd->hij", q[lo:hi], k[lo:hi]) / math.sqrt(dh)
            sc = np.where(mask[None], sc, -np.inf)
            sc = sc - sc.max(axis=2, keepdims=True)
            P = np.exp(sc)
            P = P / P.sum(axis=2, keepdims=True)
            a[lo:hi] = np.einsum("hij,jhd->ihd", P, v[lo:hi])
            Ps.append(P)
        a = a.reshape(n, db)
        x_mid = x_in + (a @ p["w_o"].T + p["b_o"])
        u2 = layer_norm(x_mid, p["ln2_g"], p["ln2_b"], eps)
        pre = u2 @ p["w_fc1"].T + p["b_fc1"]
        g = gelu(pre)
        h = x_mid + (g @ p["w_fc2"].T + p["b_fc2"])
        c.blocks.append(BlockCache(x_in, u1, q, k, v, Ps, a, x_mid, u2, pre, g))
    c.hB = h
    c.yf = layer_norm(h, wf["lnf_g"], wf["lnf_b"], eps)
    c.z = c.yf @ wf["w_out"].T + wf["b_out"]
    return c


# ------------------------------------------------------------------ Sec. 4.2: objective
def train_loss(z: np.ndarray, kv_stale: np.ndarray, kv_joint: np.ndarray, sigma_delta: np.ndarray,
               cu_seqlens: np.ndarray, cache_dtype: str) -> Tuple[float, np.ndarray]:
    """Mean over requests of 1/(N D) sum ||z - (joint - stale)/sigma_Delta||^2 (R21),
    and its gradient with respect to z."""
    tgt = (dtype_to_f64(kv_joint, cache_dtype) - dtype_to_f64(kv_stale, cache_dtype)) \
        / np.asarray(sigma_delta, np.float64)[None, :]
    r = z - tgt
    n_req = len(cu_seqlens) - 1
    D = z.shape[1]
    loss = 0.0
    dz = np.empty_like(z)
    for q in range(n_req):
        lo, hi = int(cu_seqlens[q]), int(cu_seqlens[q + 1])
        nd = (hi - lo) * D
        loss += float(np.sum(r[lo:hi] ** 2)) / nd / n_req
        dz[lo:hi] = 2.0 * r[lo:hi] / nd / n_req
    return loss, dz


# ------------------------------------------------------------------ backward, step by step in reverse
def _layer_norm_backward(x: np.ndarray, gamma: np.ndarray, dy: np.ndarray, eps: float):
    """y = (x - mean) / sqrt(var + eps) * gamma + beta (biased var): returns dx, dgamma, dbeta."""
    mu = x.mean(axis=-1, keepdims=True)
    rstd = 1.0 / np.sqrt(((x - mu) ** 2).mean(axis=-1, keepdims=True) + eps)
    xh = (x - mu) * rstd
    dxh = dy * gamma
    dx = rstd * (dxh - dxh.mean(axis=-1, keepdims=True) - xh * (dxh * xh).mean(axis=-1, keepdims=True))
    return dx, (dy * xh).sum(axis=0), dy.sum(axis=0)


def _gelu_grad(x: np.ndarray) -> np.ndarray:
    """d/dx [x Phi(x)] = Phi(x) + x phi(x)."""
    Phi = 0.5 * torch.erfc(torch.from_numpy(-x / math.sqrt(2.0))).numpy()
    return Phi + x * np.exp(-0.5 * x * x) / math.sqrt(2.0 * math.pi)


def train_backward(c: TrainCache, dz: np.ndarray, wf: Dict[str, np.ndarray], pos: np.ndarray,
                   cu_seqlens: np.ndarray, emb64: np.ndarray, *, head_dim: int, n_heads: int,
                   eps: float = 1e-5, rope_theta: float = 1e4) -> Dict[str, np.ndarray]:
    """Gradients of the loss with respect to every trained tensor (chain rule of the
    forward above, in reverse)."""
    gr: Dict[str, np.ndarray] = {}
    n = dz.shape[0]
    # head: z = W_out y_f + b_out
    gr["w_out"] = dz.T @ c.yf
    gr["b_out"] = dz.sum(axis=0)
    dyf = dz @ wf["w_out"]
    dh, gr["lnf_g"], gr["lnf_b"] = _layer_norm_backward(c.hB, wf["lnf_g"], dyf, eps)
    B = len(c.blocks)
    db = c.h0.shape[1]
    dhd = db // n_heads
    f = repair_inv_freq(dhd, rope_theta)
    scale = 1.0 / math.sqrt(dhd)
    ds = np.zeros_like(c.s)
    dW_rein = np.zeros_like(wf["w_rein"])
    db_rein = np.zeros_like(wf["b_rein"])
    for b in reversed(range(B)):
        bc = c.blocks[b]
        p = {k: wf[f"blk{b}.{k}"] for k in BLOCK}
        pre_ = f"blk{b}."
        # h = x_mid + W_fc2 g + b_fc2,  g = GELU(pre),  pre = W_fc1 u2 + b_fc1,  u2 = LN2(x_mid)
        gr[pre_ + "w_fc2"] = dh.T @ bc.g
        gr[pre_ + "b_fc2"] = dh.sum(axis=0)
        dpre = (dh @ p["w_fc2"]) * _gelu_grad(bc.pre)
        gr[pre_ + "w_fc1"] = dpre.T @ bc.u2
        gr[pre_ + "b_fc1"] = dpre.sum(axis=0)
        dx_ln, gr[pre_ + "ln2_g"], gr[pre_ + "ln2_b"] = _layer_norm_backward(
            bc.x_mid, p["ln2_g"], dpre @ p["w_fc1"], eps)
        dx_mid = dh + dx_ln
        # x_mid = x_in + W_o a + b_o
        gr[pre_ + "w_o"] = dx_mid.T @ bc.a
        gr[pre_ + "b_o"] = dx_mid.sum(axis=0)
        da = (dx_mid @ p["w_o"]).reshape(n, n_heads, dhd)
        # a = softmax(q k^T scale, masked) v per request and head
        dq = np.zeros_like(bc.q)
        dk = np.zeros_like(bc.k)
        dv = np.zeros_like(bc.v)
        for r in range(len(cu_seqlens) - 1):
            lo, hi = int(cu_seqlens[r]), int(cu_seqlens[r + 1])
            P = bc.P[r]                                                   # [h, i, j]
            dv[lo:hi] = np.einsum("hij,ihd->jhd", P, da[lo:hi])
            dP = np.einsum("ihd,jhd->hij", da[lo:hi], bc.v[lo:hi])
            dS = P * (dP - (P * dP).sum(axis=2, keepdims=True))
            dq[lo:hi] = np.einsum("hij,jhd->ihd", dS, bc.k[lo:hi]) * scale
            dk[lo:hi] = np.einsum("hij,ihd->jhd", dS, bc.q[lo:hi]) * scale
        # the repairer RoPE is a rotation: its transpose rotates back
        dq = rope_rotate_half(dq, -np.asarray(pos, np.float64), f).reshape(n, db)
        dk = rope_rotate_half(dk, -np.asarray(pos, np.float64), f).reshape(n, db)
        dqkv = np.concatenate([dq, dk, dv.reshape(n, db)], axis=1)
        gr[pre_ + "w_qkv"] = dqkv.T @ bc.u1
        gr[pre_ + "b_qkv"] = dqkv.sum(axis=0)
        dx_ln, gr[pre_ + "ln1_g"], gr[pre_ + "ln1_b"] = _layer_norm_backward(
            bc.x_in, p["ln1_g"], dqkv @ p["w_qkv"], eps)
        dx_in = dx_mid + dx_ln
        # x_in = h^{b-1} + W_rein,b s + b_rein,b
        dW_rein[b] = dx_in.T @ c.s
        db_rein[b] = dx_in.sum(axis=0)
        ds += dx_in @ wf["w_rein"][b]
        dh = dx_in
    gr["w_rein"], gr["b_rein"] = dW_rein, db_rein
    # h0 = W_fuse [s; e] + b_fuse,  e = W_tok emb + b_tok
    se = np.concatenate([c.s, c.e], axis=1)
    gr["w_fuse"] = dh.T @ se
    gr["b_fuse"] = dh.sum(axis=0)
    dse = dh @ wf["w_fuse"]
    dc = c.s.shape[1]
    ds += dse[:, :dc]
    de = dse[:, dc:]
    gr["w_tok"] = de.T @ emb64
    gr["b_tok"] = de.sum(axis=0)
    # s = W_map y + b_map,  y_{t,s} = W_seg,s x_{t,s} + b_seg,s
    gr["w_map"] = ds.T @ c.y
    gr["b_map"] = ds.sum(axis=0)
    dy = ds @ wf["w_map"]
    S = wf["w_seg"].shape[0]
    dys = dy.reshape(n, S, -1)
    gr["w_seg"] = np.einsum("tsi,tsj->sij", dys, c.x.reshape(n, S, head_dim))
    gr["b_seg"] = dys.sum(axis=0)
    return gr


# ------------------------------------------------------------------ App. A: clipping, AdamW, schedule
@dataclass
class AdamWHyper:
    beta1: float = 0.9
    beta2: float = 0.95
    weight_decay: float = 0.01
    eps: float = 1e-8
    max_norm: float = 1.0


def grad_global_norm(grads: Dict[str, np.ndarray]) -> float:
    return math.sqrt(sum(float(np.sum(np.asarray(g, np.float64) ** 2)) for g in grads.values()))


def clip_grads(grads: Dict[str, np.ndarray], max_norm: float = 1.0):
    """Global-norm clipping (R22); returns the clipped gradients and the norm before."""
    norm = grad_global_norm(grads)
    coef = min(1.0, max_norm / (norm + 1e-6))
    return {k: g * coef for k, g in grads.items()}, norm


def adamw_update(params, grads, m, v, step: int, lr: float, hp: AdamWHyper):
    """One AdamW update (R23) of every tensor; step is 1-based.  Returns new (params, m, v)."""
    out_p, out_m, out_v = {}, {}, {}
    bc1 = 1.0 - hp.beta1 ** step
    bc2 = 1.0 - hp.beta2 ** step
    for k, g in grads.items():
        th = np.asarray(params[k], np.float64) * (1.0 - lr * hp.weight_decay)
        mk = hp.beta1 * np.asarray(m[k], np.float64) + (1.0 - hp.beta1) * g
        vk = hp.beta2 * np.asarray(v[k], np.float64) + (1.0 - hp.beta2) * g * g
        m_hat, v_hat = mk / bc1, vk / bc2
        out_p[k] = th - lr * m_hat / (np.sqrt(v_hat) + hp.eps)
        out_m[k], out_v[k] = mk, vk
    return out_p, out_m, out_v


def lr_schedule(step: int, *, peak: float = 3e-4, final: float = 3e-5, warmup: int = 2000,
                total: int = 100000) -> float:
    """R24: linear warmup to the peak, then cosine decay to the final rate."""
    if step <= warmup:
        return peak * step / warmup
    frac = min(1.0, (step - warmup) / max(1, total - warmup))
    return final + 0.5 * (peak - final) * (1.0 + math.cos(math.pi * frac))


def train_step(params, m, v, step: int, lr: float, batch: Dict[str, np.ndarray], *, sigma_stale,
               sigma_delta, cache_dtype: str, head_dim: int, n_heads: int, hp: AdamWHyper = AdamWHyper(),
               eps: float = 1e-5, rope_theta: float = 1e4, mask_mode: str = "block_causal"):
    """Forward, loss, backward, clipping and AdamW: one update.  batch holds the
    assembled stale cache, the joint cache, embeddings, chunk_id, pos and cu_seqlens.
    Returns (loss, grad norm, raw grads, new params, new m, new v)."""
    wf = forward_weights(params)
    wf["sigma_stale"], wf["sigma_delta"] = sigma_stale, sigma_delta
    c = train_forward(batch["kv"], batch["emb"], batch["chunk_id"], batch["pos"], batch["cu_seqlens"],
                      wf, cache_dtype=cache_dtype, head_dim=head_dim, n_heads=n_heads, eps=eps,
                      rope_theta=rope_theta, mask_mode=mask_mode)
    loss, dz = train_loss(c.z, batch["kv"], batch["kv_joint"], sigma_delta, batch["cu_seqlens"],
                          cache_dtype)
    grads = train_backward(c, dz, wf, batch["pos"], batch["cu_seqlens"],
                           dtype_to_f64(batch["emb"], cache_dtype), head_dim=head_dim,
                           n_heads=n_heads, eps=eps, rope_theta=rope_theta)
    clipped, norm = clip_grads(grads, hp.max_norm)
    new_p, new_m, new_v = adamw_update(params, clipped, m, v, step, lr, hp)
    return loss, norm, grads, new_p, new_m, new_v
