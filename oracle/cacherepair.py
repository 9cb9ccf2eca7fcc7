"""Oracle: the CacheRepair online repair forward, written out plainly in float64.

TEST INFRASTRUCTURE.  This module is the slow, obviously-correct statement of
what the GPU library computes.  It is imported only by the tests, the smoke
check and the CPU-baseline legs of the benchmark; the product path never
imports it and shares no code with it.  Matrix products use numpy's matmul
(a library primitive); everything else is the paper's definition, in the
paper's order, in float64 on values read exactly from the stored inputs.

Paper: "CacheRepair: Learning to Repair Cross-Chunk Context in RAG for KV
Cache Fusion" (arxiv 2609.35139).  Section references are to that paper:
  Sec. 2.2  Problem setting: stale cache, R_theta(KV_stale, D_r) ~ KV_joint.
  Sec. 4.1  Inference: canonical chunk caches; StaleEncoder and token fusion;
            Repair Blocks with the block-causal mask and stale-feature
            reinjection; LN + KV residual head; residual add; global RoPE on K.
  App. A    Repairer configurations: 64-dim attention heads, MLP ratio 3
            (Table "repair-scales").
  App. D    Parameter allocation (Table "repair-parameter-groups"); the head
            is affine, b + col(W_out).
  App. I    Cache payload 2 N D_KV bytes (bf16).

Readings where the paper is silent:
  R1  Widths: the StaleEncoder and P_tok output width d_c; F: 2 d_c -> d_b;
      P_b: d_c -> d_b; backbone and head at d_b.  With d_c = d_b this is the
      paper's single width.
  R3  No nonlinearity inside the StaleEncoder (two affine maps, kept separate).
  R4  Repair Block = pre-LN residual block: x + Attn(LN1 x), then
      x + MLP(LN2 x); LayerNorm affine, biased variance, eps 1e-5; MLP is
      Linear -> erf-GELU -> Linear; every linear has a bias.
  R6  Repairer RoPE: base 1e4, rotate-half pairs (i, i + d/2) over the whole
      head, angle = p_t * base^(-2i/d), p_t = position in the request.
  R7  Attention scale 1/sqrt(d_head); token i sees j iff c(j) <= c(i)
      (self included); attention never crosses requests.
  R9  D_KV coordinate j = ((layer*2 + kv)*H + head)*d_h + d, kv = 0 for K;
      segment s is the slice [s*d_h, (s+1)*d_h).
  R10 Global RoPE (target R_M) applied after the residual add, rotate-half
      pairs within each K segment, frequencies supplied by the caller.
  R11 The repaired value is formed exactly, then rounded once to the cache
      dtype (round to nearest even for bf16).
  R18 The attention-topology variants of App. F change only the mask:
      A1 "strict token-causal" is j <= i (self included, as in R7), A2 is
      every token of the request, A3 "block-diagonal" is c(j) == c(i).
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Dict, List, Optional, Sequence

import numpy as np
import torch

__all__ = [
    "dtype_to_f64", "round_to_cache", "assemble_stale", "segment_projection", "stale_encoder", "token_fusion",
    "reinjection", "layer_norm", "gelu", "rope_rotate_half", "block_causal_mask",
    "block_causal_attention", "repair_block", "repair_backbone", "residual_head",
    "apply_residual", "global_rope_k", "repair_request", "weight_shapes", "param_groups",
    "cache_payload_bytes", "OracleResult", "repair_inv_freq", "block_weights",
    "MASK_MODES", "attention_mask", "masked_attention",
]


# ------------------------------------------------------------------ numbers
def dtype_to_f64(x: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 value of stored cache/weight data (bf16 bit patterns or fp32)."""
    if dtype == "f32" or x.dtype == np.float32:
        return np.asarray(x, dtype=np.float64)
    assert x.dtype == np.uint16, x.dtype
    return ((x.astype(np.uint32) << 16).view(np.float32)).astype(np.float64)


def round_to_cache(x: np.ndarray, dtype: str) -> np.ndarray:
    """Round exact values once to the cache dtype (R11).

    fp32: IEEE round-to-nearest-even of the float64 value.
    bf16: round-to-nearest-even of the float64 value to 8 significant bits,
    done in integer arithmetic on the float64 bit pattern (so there is no
    intermediate rounding through fp32).  Returns fp32 or uint16 bits.
    """
    if dtype == "f32":
        return x.astype(np.float32)
    x = np.asarray(x, dtype=np.float64)
    bits = x.view(np.uint64)
    sign = (bits >> np.uint64(63)).astype(np.uint16) << np.uint16(15)
    a = np.abs(x)
    # bf16 keeps 7 explicit mantissa bits; float64 has 52 -> drop 45 bits.
    ab = a.view(np.uint64)
    drop = np.uint64(45)
    half = np.uint64(1) << (drop - np.uint64(1))
    mask = (np.uint64(1) << drop) - np.uint64(1)
    rem = ab & mask
    q = ab >> drop
    up = (rem > half) | ((rem == half) & ((q & np.uint64(1)) == np.uint64(1)))
    q = q + up.astype(np.uint64)
    # q is now the rounded value's top bits of the float64 encoding:
    # 11-bit exponent + 7-bit mantissa.  Re-bias the exponent to bf16's 8 bits.
    exp64 = (q >> np.uint64(7)).astype(np.int64)
    man = (q & np.uint64(0x7F)).astype(np.int64)
    exp32 = exp64 - 1023 + 127
    out = np.zeros(x.shape, np.uint16)
    normal = (exp32 > 0) & (exp32 < 255) & (a > 0)
    out[normal] = ((exp32[normal] << 7) | man[normal]).astype(np.uint16)
    # Values this path produces are far from the bf16 range limits; anything
    # outside the normal range is flagged loudly rather than handled.
    if np.any((a > 0) & ~normal):
        raise OverflowError("value outside the bf16 normal range")
    return out | sign * (out != 0)


def _bf16_mat(w: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float64; float arrays (already converted) pass through."""
    if w.dtype == np.uint16:
        return dtype_to_f64(w, "bf16")
    return np.asarray(w, dtype=np.float64)


def _vec(v: np.ndarray) -> np.ndarray:
    return np.asarray(v, dtype=np.float64)


# ------------------------------------------------------------------ Sec. 2.2 / 4.1: assembly
def assemble_stale(kv_pool: np.ndarray, emb_pool: np.ndarray, chunk_start: np.ndarray,
                   chunk_len: np.ndarray, chunk_idx: np.ndarray, cu_chunks: np.ndarray) -> Dict:
    """Concatenate the selected canonical chunk caches in document order (Sec. 4.1).

    Canonical K carries no RoPE, so assembly is a pure copy (the paper's
    re-rotation of Sec. 2.2 belongs to the stale-only baseline; the method
    applies global RoPE after repair).  Per request r with chunks
    chunk_idx[cu_chunks[r]:cu_chunks[r+1]]:
      chunk_id[t]  = index of t's chunk within its request (c(t), Sec. 4.1)
      chunk_end[t] = exclusive end (request-local) of t's chunk
      pos[t]       = t's position in its request (p_t, Sec. 4.1)
    """
    kv_rows, emb_rows, cid, cend, pos = [], [], [], [], []
    cu_seq = [0]
    for r in range(len(cu_chunks) - 1):
        t = 0
        for k, c in enumerate(chunk_idx[cu_chunks[r]:cu_chunks[r + 1]]):
            a, n = int(chunk_start[c]), int(chunk_len[c])
            kv_rows.append(kv_pool[a:a + n])
            emb_rows.append(emb_pool[a:a + n])
            cid += [k] * n
            cend += [t + n] * n
            pos += list(range(t, t + n))
            t += n
        cu_seq.append(cu_seq[-1] + t)
    return dict(kv=np.concatenate(kv_rows), emb=np.concatenate(emb_rows),
                chunk_id=np.asarray(cid, np.int32), chunk_end=np.asarray(cend, np.int32),
                pos=np.asarray(pos, np.int32), cu_seqlens=np.asarray(cu_seq, np.int32))


# ------------------------------------------------------------------ Sec. 4.1: StaleEncoder, fusion
def segment_projection(kv: np.ndarray, sigma_stale: np.ndarray, w_seg: np.ndarray,
                       b_seg: np.ndarray, head_dim: int,
                       cache_dtype: Optional[str] = None) -> np.ndarray:
    """StaleEncoder stage 1 (Sec. 4.1): y[t, s] = W_seg,s (kv_t,s / sigma_stale,s) + b_seg,s.

    kv: [n, D_KV] (float64, or the stored cache with `cache_dtype`); segment s
    is the slice [s d_h, (s+1) d_h) (R9).  Returns [n, S * d_seg], the S
    outputs concatenated in segment order.
    """
    x = dtype_to_f64(kv, cache_dtype) if cache_dtype else kv
    n = x.shape[0]
    S = x.shape[1] // head_dim
    W = _bf16_mat(w_seg)                                         # [S, d_seg, d_h]
    x = (x / _vec(sigma_stale)[None, :]).reshape(n, S, head_dim)
    y = np.matmul(x.transpose(1, 0, 2), W.transpose(0, 2, 1)).transpose(1, 0, 2)
    return (y + _vec(b_seg)[None]).reshape(n, -1)


def stale_encoder(kv: np.ndarray, sigma_stale: np.ndarray, w_seg: np.ndarray, b_seg: np.ndarray,
                  w_map: np.ndarray, b_map: np.ndarray, head_dim: int,
                  cache_dtype: Optional[str] = None, rows_per_step: int = 256) -> np.ndarray:
    """s_t = StaleEncoder(KV^c_stale,t / sigma_stale)  (Sec. 4.1).

    Stage 1 (`segment_projection`): one d_h -> d_seg linear per segment on the
    cache divided by sigma_stale; stage 2: the concatenated S outputs mapped
    to d_c (R1, R3).  Tokens are independent, so they are processed
    `rows_per_step` at a time to bound memory.
    """
    n = kv.shape[0]
    W = _bf16_mat(w_seg)
    Wm = _bf16_mat(w_map)
    out = np.empty((n, Wm.shape[0]))
    for a in range(0, n, rows_per_step):
        y = segment_projection(kv[a:a + rows_per_step], sigma_stale, W, b_seg, head_dim,
                               cache_dtype)
        out[a:a + rows_per_step] = y @ Wm.T + _vec(b_map)
    return out


def token_fusion(s: np.ndarray, emb: np.ndarray, w_tok, b_tok, w_fuse, b_fuse) -> np.ndarray:
    """h^0_t = F([s_t ; P_tok E_M(x_t)])  (Sec. 4.1), F and P_tok affine."""
    e = emb @ _bf16_mat(w_tok).T + _vec(b_tok)
    return np.concatenate([s, e], axis=1) @ _bf16_mat(w_fuse).T + _vec(b_fuse)


def reinjection(s: np.ndarray, w_rein_b, b_rein_b) -> np.ndarray:
    """P_b(s): the block-b projection of the encoded features (Sec. 4.1)."""
    return s @ _bf16_mat(w_rein_b).T + _vec(b_rein_b)


# ------------------------------------------------------------------ Sec. 4.1: Repair Block parts
def layer_norm(x: np.ndarray, g, b, eps: float) -> np.ndarray:
    """LayerNorm over the last axis: biased variance, affine (R4)."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * _vec(g) + _vec(b)


def gelu(x: np.ndarray) -> np.ndarray:
    """erf-form GELU, x * Phi(x) (R4)."""
    return 0.5 * x * (1.0 + torch.erf(torch.from_numpy(x / math.sqrt(2.0))).numpy())


def rope_rotate_half(x: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray) -> np.ndarray:
    """Rotate pairs (i, i + d/2) of the last axis by angle pos * inv_freq[i].

    x: [N, ..., d]; pos: [N]; inv_freq: [d/2].  Used for the repairer's own
    RoPE on Q and K (Sec. 4.1, R6) and for the target's R_M (R10).
    """
    d = x.shape[-1]
    h = d // 2
    ang = pos.astype(np.float64)[:, None] * _vec(inv_freq)[None, :]      # [N, d/2]
    shape = (x.shape[0],) + (1,) * (x.ndim - 2) + (h,)
    c, s = np.cos(ang).reshape(shape), np.sin(ang).reshape(shape)
    a, b = x[..., :h], x[..., h:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def block_causal_mask(chunk_id: np.ndarray) -> np.ndarray:
    """A_ij = 1[c(j) <= c(i)]  (Sec. 4.1, block-causal mask)."""
    return chunk_id[None, :] <= chunk_id[:, None]


def block_causal_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray,
                           chunk_id: np.ndarray) -> np.ndarray:
    """Multi-head softmax attention under the block-causal mask, one request.

    q, k, v: [N, n_heads, d_head] (RoPE already applied to q, k).  Query i
    attends to the keys j with c(j) <= c(i) (R7).  Chunk ids are
    non-decreasing along the request, so for every query of chunk c that set
    is the prefix of tokens up to the end of chunk c; the softmax
    (max-subtracted) of q k^T / sqrt(d_head) is taken over exactly that set.
    """
    n, nh, dh = q.shape
    out = np.empty_like(q)
    assert np.all(np.diff(chunk_id) >= 0), "chunk ids must be non-decreasing"
    for c in np.unique(chunk_id):
        rows = np.nonzero(chunk_id == c)[0]
        end = int(np.nonzero(chunk_id <= c)[0].max()) + 1      # keys j with c(j) <= c
        for h in range(nh):
            sc = (q[rows, h, :] @ k[:end, h, :].T) / math.sqrt(dh)
            sc = sc - sc.max(axis=1, keepdims=True)
            p = np.exp(sc)
            p = p / p.sum(axis=1, keepdims=True)
            out[rows, h, :] = p @ v[:end, h, :]
    return out


MASK_MODES = ("block_causal", "token_causal", "bidirectional", "block_diagonal")


def attention_mask(chunk_id: np.ndarray, mode: str) -> np.ndarray:
    """A[i, j] = True iff query i attends to key j, one request.

    block_causal   c(j) <= c(i)   the method's mask (Sec. 4.1), ablation A0
    token_causal   j <= i         ablation A1 (App. F, R18)
    bidirectional  every j        ablation A2 (App. F)
    block_diagonal c(j) == c(i)   ablation A3 (App. F, R18)
    """
    n = len(chunk_id)
    ci, cj = chunk_id[:, None], chunk_id[None, :]
    i, j = np.arange(n)[:, None], np.arange(n)[None, :]
    if mode == "block_causal":
        return cj <= ci
    if mode == "token_causal":
        return j <= i
    if mode == "bidirectional":
        return np.ones((n, n), bool)
    if mode == "block_diagonal":
        return cj == ci
    raise ValueError(f"unknown mask mode {mode!r}")


def masked_attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, mask: np.ndarray) -> np.ndarray:
    """Multi-head softmax attention of one request under an explicit mask.

    q, k, v: [N, n_heads, d_head]; mask: [N, N] bool, every row with at least
    one True.  Per head, the full score matrix q k^T / sqrt(d_head) is formed,
    entries outside the mask are set to -inf, and each row's softmax
    (max-subtracted) weights the values.
    """
    n, nh, dh = q.shape
    assert mask.shape == (n, n) and mask.any(axis=1).all(), "every query needs a visible key"
    out = np.empty_like(q)
    for h in range(nh):
        sc = (q[:, h, :] @ k[:, h, :].T) / math.sqrt(dh)
        sc = np.where(mask, sc, -np.inf)
        sc = sc - sc.max(axis=1, keepdims=True)
        p = np.exp(sc)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, h, :] = p @ v[:, h, :]
    return out


def repair_inv_freq(head_dim: int, theta: float) -> np.ndarray:
    i = np.arange(head_dim // 2, dtype=np.float64)
    return theta ** (-2.0 * i / head_dim)


def repair_block(x: np.ndarray, blk: Dict[str, np.ndarray], chunk_id: np.ndarray,
                 pos: np.ndarray, n_heads: int, eps: float, rope_theta: float,
                 mask_mode: str = "block_causal") -> np.ndarray:
    """One Repair Block: attention then MLP, pre-LN residual form (Sec. 4.1, R4).

    x is the block input h^{b-1} + P_b(s).  `mask_mode` selects the attention
    topology (App. F); the default is the method's block-causal mask.
    """
    n, db = x.shape
    dh = db // n_heads
    u = layer_norm(x, blk["ln1_g"], blk["ln1_b"], eps)
    qkv = u @ _bf16_mat(blk["w_qkv"]).T + _vec(blk["b_qkv"])
    q = qkv[:, :db].reshape(n, n_heads, dh)
    k = qkv[:, db:2 * db].reshape(n, n_heads, dh)
    v = qkv[:, 2 * db:].reshape(n, n_heads, dh)
    f = repair_inv_freq(dh, rope_theta)
    q, k = rope_rotate_half(q, pos, f), rope_rotate_half(k, pos, f)
    if mask_mode == "block_causal":
        a = block_causal_attention(q, k, v, chunk_id).reshape(n, db)
    else:
        a = masked_attention(q, k, v, attention_mask(chunk_id, mask_mode)).reshape(n, db)
    x = x + (a @ _bf16_mat(blk["w_o"]).T + _vec(blk["b_o"]))
    u = layer_norm(x, blk["ln2_g"], blk["ln2_b"], eps)
    g = gelu(u @ _bf16_mat(blk["w_fc1"]).T + _vec(blk["b_fc1"]))
    return x + (g @ _bf16_mat(blk["w_fc2"]).T + _vec(blk["b_fc2"]))


def block_weights(w: Dict[str, np.ndarray], b: int) -> Dict[str, np.ndarray]:
    p = f"blk{b}."
    return {k[len(p):]: v for k, v in w.items() if k.startswith(p)}


def repair_backbone(h0: np.ndarray, s: np.ndarray, w: Dict[str, np.ndarray],
                    chunk_id: np.ndarray, pos: np.ndarray, n_heads: int, eps: float,
                    rope_theta: float, keep: Optional[List] = None,
                    mask_mode: str = "block_causal") -> np.ndarray:
    """h^b = RepairBlock_b(h^{b-1} + P_b(s); A, p), b = 1..B  (Sec. 4.1)."""
    h = h0
    for b in range(w["w_rein"].shape[0]):
        h = repair_block(h + reinjection(s, w["w_rein"][b], w["b_rein"][b]),
                         block_weights(w, b), chunk_id, pos, n_heads, eps, rope_theta,
                         mask_mode=mask_mode)
        if keep is not None:
            keep.append(h)
    return h


# ------------------------------------------------------------------ Sec. 4.1: head, residual, R_M
def residual_head(hB: np.ndarray, lnf_g, lnf_b, w_out, b_out, eps: float,
                  cols: Optional[np.ndarray] = None) -> np.ndarray:
    """z_t = KVResidualHead(LN(h^B_t)), the head affine: W_out y + b_out (Sec. 4.1, App. D).

    `cols` optionally restricts the output to a subset of D_KV coordinates.
    """
    y = layer_norm(hB, lnf_g, lnf_b, eps)
    W = _bf16_mat(w_out if cols is None else w_out[cols])
    b = _vec(b_out if cols is None else np.asarray(b_out)[cols])
    return y @ W.T + b


def apply_residual(kv: np.ndarray, z: np.ndarray, sigma_delta: np.ndarray) -> np.ndarray:
    """KV^c_repair = KV^c_stale + sigma_Delta (elementwise) z  (Sec. 4.1), exact."""
    return kv + _vec(sigma_delta)[None, :] * z


def global_rope_k(kvhat: np.ndarray, pos: np.ndarray, inv_freq: np.ndarray, n_layers: int,
                  n_kv_heads: int, head_dim: int) -> np.ndarray:
    """K_repair = R_M(p_t) K^c_repair, V unchanged (Sec. 4.1, R9, R10)."""
    n = kvhat.shape[0]
    x = kvhat.reshape(n, n_layers, 2, n_kv_heads, head_dim).copy()
    x[:, :, 0] = rope_rotate_half(x[:, :, 0], pos, inv_freq)
    return x.reshape(n, -1)


# ------------------------------------------------------------------ whole request
@dataclass
class OracleResult:
    s: np.ndarray
    h0: np.ndarray
    rein: List[np.ndarray]
    blocks: List[np.ndarray]
    yf: np.ndarray
    z: Optional[np.ndarray]
    repaired: Optional[np.ndarray]        # exact (float64), canonical K (before R_M)
    repaired_rot: Optional[np.ndarray]    # exact (float64), after R_M on K


def repair_request(kv: np.ndarray, emb: np.ndarray, chunk_id: np.ndarray, pos: np.ndarray,
                   w: Dict[str, np.ndarray], *, cache_dtype: str, n_layers: int, n_kv_heads: int,
                   head_dim: int, n_heads: int, eps: float = 1e-5, rope_theta: float = 1e4,
                   inv_freq_target: Optional[np.ndarray] = None, with_head: bool = True,
                   head_cols: Optional[np.ndarray] = None,
                   mask_mode: str = "block_causal") -> OracleResult:
    """The full repair forward of one request (Sec. 4.1), all in float64.

    kv/emb are the assembled stale cache and embeddings in their stored
    dtype; the result's `repaired` is the exact repaired cache, to be
    rounded with `round_to_cache` for a bit-level comparison.
    """
    w = {k_: (_bf16_mat(v_) if v_.dtype == np.uint16 else v_) for k_, v_ in w.items()}
    emb64 = dtype_to_f64(emb, cache_dtype)
    s = stale_encoder(kv, w["sigma_stale"], w["w_seg"], w["b_seg"], w["w_map"], w["b_map"],
                      head_dim, cache_dtype=cache_dtype)
    h0 = token_fusion(s, emb64, w["w_tok"], w["b_tok"], w["w_fuse"], w["b_fuse"])
    rein = [reinjection(s, w["w_rein"][b], w["b_rein"][b]) for b in range(w["w_rein"].shape[0])]
    blocks: List[np.ndarray] = []
    hB = repair_backbone(h0, s, w, chunk_id, pos, n_heads, eps, rope_theta, keep=blocks,
                         mask_mode=mask_mode)
    yf = layer_norm(hB, w["lnf_g"], w["lnf_b"], eps)
    z = rep = rot = None
    if with_head:
        z = residual_head(hB, w["lnf_g"], w["lnf_b"], w["w_out"], w["b_out"], eps, cols=head_cols)
        kv64 = dtype_to_f64(kv if head_cols is None else kv[:, head_cols], cache_dtype)
        base = kv64
        sd = w["sigma_delta"] if head_cols is None else w["sigma_delta"][head_cols]
        rep = apply_residual(base, z, sd)
        if inv_freq_target is not None and head_cols is None:
            rot = global_rope_k(rep, pos, inv_freq_target, n_layers, n_kv_heads, head_dim)
    return OracleResult(s, h0, rein, blocks, yf, z, rep, rot)


# ------------------------------------------------------------------ shapes and sizes
def weight_shapes(n_layers: int, n_kv_heads: int, head_dim: int, d_model: int, d_seg: int,
                  d_c: int, d_b: int, n_blocks: int, mlp_hidden: int) -> Dict[str, tuple]:
    """Every trainable tensor of the repairer, by the group App. D reports it in."""
    S = 2 * n_layers * n_kv_heads
    D = S * head_dim
    g: Dict[str, tuple] = {
        "encoder.w_seg": (S, d_seg, head_dim), "encoder.b_seg": (S, d_seg),
        "encoder.w_map": (d_c, S * d_seg), "encoder.b_map": (d_c,),
        "fusion.w_tok": (d_c, d_model), "fusion.b_tok": (d_c,),
        "fusion.w_fuse": (d_b, 2 * d_c), "fusion.b_fuse": (d_b,),
        "reinjection.w_rein": (n_blocks, d_b, d_c), "reinjection.b_rein": (n_blocks, d_b),
        "head.w_out": (D, d_b), "head.b_out": (D,),
    }
    for b in range(n_blocks):
        g.update({
            f"backbone.blk{b}.ln1_g": (d_b,), f"backbone.blk{b}.ln1_b": (d_b,),
            f"backbone.blk{b}.w_qkv": (3 * d_b, d_b), f"backbone.blk{b}.b_qkv": (3 * d_b,),
            f"backbone.blk{b}.w_o": (d_b, d_b), f"backbone.blk{b}.b_o": (d_b,),
            f"backbone.blk{b}.ln2_g": (d_b,), f"backbone.blk{b}.ln2_b": (d_b,),
            f"backbone.blk{b}.w_fc1": (mlp_hidden, d_b), f"backbone.blk{b}.b_fc1": (mlp_hidden,),
            f"backbone.blk{b}.w_fc2": (d_b, mlp_hidden), f"backbone.blk{b}.b_fc2": (d_b,),
        })
    g["backbone.lnf_g"] = (d_b,)
    g["backbone.lnf_b"] = (d_b,)
    return g


def param_groups(**dims) -> Dict[str, int]:
    """Parameter count per App. D group (encoder, fusion, reinjection, backbone, head, total)."""
    out: Dict[str, int] = {}
    for name, shp in weight_shapes(**dims).items():
        grp = name.split(".")[0]
        out[grp] = out.get(grp, 0) + int(np.prod(shp))
    out["total"] = sum(out.values())
    return out


def cache_payload_bytes(n_tokens: int, n_layers: int, n_kv_heads: int, head_dim: int,
                        bytes_per_elem: int = 2) -> int:
    """Stale/repaired cache size: N * D_KV elements, D_KV = 2 L H_kv d_h (App. I)."""
    return n_tokens * 2 * n_layers * n_kv_heads * head_dim * bytes_per_elem
