"""RepairSession: device buffers for one GPU and the four-call repair chain.

A user of the library creates a session for a target/repairer shape and a
token capacity, then calls ``repair()`` per batch of requests.  Everything
computed runs in the library's kernels through the C ABI; this class only
owns buffers (torch allocations) and passes pointers.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import Dict, Optional

import numpy as np
import torch

from . import cr


def _dtype(cache_dtype: int) -> torch.dtype:
    return torch.float32 if cache_dtype == cr.CR_F32 else torch.bfloat16


@dataclass
class Assembled:
    n_tokens: int
    cu_seqlens: np.ndarray       # host int32 [n_req + 1]


class RepairSession:
    def __init__(self, target: cr.cr_target_dims, rep: cr.cr_repairer_dims,
                 weights: cr.PackedWeights, max_tokens: int, device="cuda"):
        self.target, self.rep, self.weights = target, rep, weights
        self.device = torch.device(device)
        S = 2 * target.n_layers * target.n_kv_heads
        self.d_kv = S * target.head_dim
        dt = _dtype(target.cache_dtype)
        n = max_tokens
        z = lambda *shape, dtype: torch.empty(*shape, dtype=dtype, device=self.device)
        self.kv = z(n, self.d_kv, dtype=dt)
        self.emb = z(n, target.d_model, dtype=dt)
        self.chunk_id = z(n, dtype=torch.int32)
        self.chunk_end = z(n, dtype=torch.int32)
        self.pos = z(n, dtype=torch.int32)
        self.cu_seqlens = z(257, dtype=torch.int32)
        self.h0 = z(n, rep.d_b, dtype=torch.float32)
        self.rein = z(n, max(rep.n_blocks, 1) * rep.d_b, dtype=torch.float32)
        self.yf = z(n, rep.d_b, dtype=torch.bfloat16)
        ws = cr.cr_workspace_bytes(target, rep, n)
        if ws == 0:
            raise cr.CrError("cr_workspace_bytes", cr.CR_ERR_INVALID_ARG, "invalid dimensions")
        self.workspace = z((ws + 15) // 16 * 16, dtype=torch.uint8)
        self.max_tokens = n

    # -------------------------------------------------------------- the four calls
    def assemble(self, kv_pool: torch.Tensor, emb_pool: torch.Tensor, chunk_start, chunk_len,
                 chunk_idx, cu_chunks, stream=None) -> Assembled:
        n, cu = cr.cr_assemble_stale(self.target, kv_pool, emb_pool, chunk_start, chunk_len,
                                     chunk_idx, cu_chunks, self.kv, self.emb, self.chunk_id,
                                     self.chunk_end, self.pos, self.cu_seqlens, stream)
        return Assembled(n, cu)

    def compress(self, a: Assembled, stream=None):
        cr.cr_compress_features(self.target, self.rep, self.weights, self.kv, self.emb, a.n_tokens,
                                self.h0, self.rein, self.workspace, stream)

    def assemble_compress(self, kv_pool: torch.Tensor, emb_pool: torch.Tensor, chunk_start,
                          chunk_len, chunk_idx, cu_chunks, stream=None, write_kv=True) -> Assembled:
        """assemble + compress as one call: the segment projection reads the pool and
        writes the assembled cache as it goes (same results, one cache read fewer);
        write_kv=False (bf16 caches) leaves kv unwritten, for apply_pool."""
        n, cu = cr.cr_assemble_compress(self.target, self.rep, self.weights, kv_pool, emb_pool,
                                        chunk_start, chunk_len, chunk_idx, cu_chunks,
                                        self.kv if write_kv else None, self.emb, self.chunk_id,
                                        self.chunk_end, self.pos, self.cu_seqlens, self.h0,
                                        self.rein, self.workspace, stream)
        return Assembled(n, cu)

    def forward(self, a: Assembled, stream=None, mask_mode="block_causal"):
        """The Repair Blocks and LN_f; mask_mode picks the attention mask (the method's
        block-causal mask, or an App. F ablation: token_causal, bidirectional, block_diagonal)."""
        if mask_mode in ("block_causal", cr.CR_MASK_BLOCK_CAUSAL):
            cr.cr_repair_forward(self.target, self.rep, self.weights, self.h0, self.rein,
                                 self.chunk_end, self.pos, a.cu_seqlens, a.n_tokens, self.yf,
                                 self.workspace, stream)
        else:
            cr.cr_repair_forward_masked(self.target, self.rep, self.weights, self.h0, self.rein,
                                        self.chunk_end, self.pos, a.cu_seqlens, a.n_tokens,
                                        mask_mode, self.yf, self.workspace, stream)

    def apply(self, a: Assembled, inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None,
              component="kv", offset="stale", keep_first_chunk=False):
        """Head and residual add in place on kv.  The defaults are the method; the
        output choices (App. F) repair only K or only V, drop the stale offset (A5),
        or keep each request's first chunk stale."""
        if component == "kv" and offset == "stale" and not keep_first_chunk:
            cr.cr_apply_residual(self.target, self.rep, self.weights, self.yf, a.n_tokens, self.kv,
                                 self.pos, inv_freq_target, rope_mode, workspace=self.workspace,
                                 stream=stream)
        else:
            cr.cr_apply_residual_select(self.target, self.rep, self.weights, self.yf, a.n_tokens,
                                        self.kv, self.pos, inv_freq_target, rope_mode, component,
                                        offset, self.chunk_id if keep_first_chunk else None,
                                        workspace=self.workspace, stream=stream)

    def apply_pool(self, a: Assembled, kv_pool: torch.Tensor, chunk_start, chunk_len, chunk_idx,
                   cu_chunks, inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None):
        """Head and residual add with the stale rows read from the pool (the chunk map of
        the assemble call) and the repaired rows written to kv (bf16 caches)."""
        cr.cr_apply_residual_pool(self.target, self.rep, self.weights, self.yf, a.n_tokens, kv_pool,
                                  chunk_start, chunk_len, chunk_idx, cu_chunks, self.kv, self.pos,
                                  inv_freq_target, rope_mode, workspace=self.workspace, stream=stream)

    def stale_kv(self, a: Assembled, inv_freq_target, stream=None):
        """The stale cache of independent reuse: the assembled canonical cache with K
        rotated to its request positions (no repair), in place on kv."""
        cr.cr_rotate_k(self.target, self.kv, a.n_tokens, self.pos, inv_freq_target, stream)

    def apply_paged(self, a: Assembled, slot_mapping: torch.Tensor, paged_cache: torch.Tensor,
                    num_slots: int, inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None):
        """Head and residual add with the repaired rows written to a paged target cache
        ([2 L, num_slots, H_kv d_h] bf16) at slot_mapping[t] (int64, < 0 = skip); kv stays stale."""
        cr.cr_apply_residual_paged(self.target, self.rep, self.weights, self.yf, a.n_tokens, self.kv,
                                   self.pos, slot_mapping, paged_cache, num_slots, inv_freq_target,
                                   rope_mode, workspace=self.workspace, stream=stream)

    def repair(self, kv_pool, emb_pool, chunk_start, chunk_len, chunk_idx, cu_chunks,
               inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None,
               mask_mode="block_causal", component="kv", offset="stale",
               keep_first_chunk=False) -> Assembled:
        """Assemble, compress, run the blocks and apply the residual; kv holds the result.
        The keyword options select the App. F mask and output variants (defaults: the method).
        For a bf16 cache under the method's output the stale rows never go through kv: the
        encoder and the head read them from the pool (the same results, one write and one read
        of the cache fewer)."""
        pooled = (self.target.cache_dtype == cr.CR_BF16 and component == "kv" and offset == "stale"
                  and not keep_first_chunk)
        a = self.assemble_compress(kv_pool, emb_pool, chunk_start, chunk_len, chunk_idx, cu_chunks,
                                   stream, write_kv=not pooled)
        self.forward(a, stream, mask_mode=mask_mode)
        if pooled:
            self.apply_pool(a, kv_pool, chunk_start, chunk_len, chunk_idx, cu_chunks, inv_freq_target,
                            rope_mode, stream)
        else:
            self.apply(a, inv_freq_target, rope_mode, stream, component=component, offset=offset,
                       keep_first_chunk=keep_first_chunk)
        return a


def pack_host_weights(w: Dict[str, np.ndarray], n_blocks: int, device="cuda") -> cr.PackedWeights:
    """Copy a host weight dict (bf16 bit patterns as uint16, fp32 vectors) to the device."""
    dev = {}
    for k, v in w.items():
        a = np.ascontiguousarray(v)
        if a.dtype == np.uint16:
            t = torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
        else:
            t = torch.from_numpy(a.astype(np.float32, copy=False))
        dev[k] = t.to(device)
    return cr.PackedWeights(dev, n_blocks)


def host_to_device(a: np.ndarray, device="cuda") -> torch.Tensor:
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(a).to(device)


def dims_from(target, repairer):
    """cr structs from objects with the field names of cr.h (e.g. the test fixtures)."""
    t = cr.target_dims(target.n_layers, target.n_kv_heads, target.head_dim, target.d_model,
                       target.cache_dtype)
    r = cr.repairer_dims(repairer.d_seg, repairer.d_c, repairer.d_b, repairer.n_blocks,
                         repairer.n_heads, repairer.mlp_hidden, repairer.ln_eps,
                         repairer.rope_theta)
    return t, r


class RepairPipeline:
    """Serving loop that hides host<->device transfers behind the repair.

    Requests arrive as chunk caches in pinned host memory and leave as repaired
    caches in pinned host memory.  Two slots (each a RepairSession plus a device
    staging pool) alternate: while one slot repairs request i on the compute
    stream, request i+1's chunks are copied into the other slot's staging pool
    on a host-to-device stream and request i-1's repaired cache is copied back
    on a device-to-host stream.  A slot is reused only after its previous repair
    has consumed the staging pool and its previous result has been read back,
    so the per-request time approaches the slower of the link and the repair.
    This is the copy-stream overlap of the serving integration the paper names
    as future work (Sec. 6); the paged target-cache write is not part of it.

    Only stream/event plumbing lives here: the copies are cudaMemcpyAsync calls
    (torch ``copy_``) and every step of the repair runs in the library's kernels.
    """

    def __init__(self, target: cr.cr_target_dims, rep: cr.cr_repairer_dims,
                 weights: cr.PackedWeights, max_tokens: int, device="cuda", n_slots: int = 2):
        self.device = torch.device(device)
        self.n_slots = n_slots
        self.slots = [RepairSession(target, rep, weights, max_tokens, device) for _ in range(n_slots)]
        dt = _dtype(target.cache_dtype)
        d_kv = self.slots[0].d_kv
        self.stage_kv = [torch.empty(max_tokens, d_kv, dtype=dt, device=self.device) for _ in range(n_slots)]
        self.stage_emb = [torch.empty(max_tokens, target.d_model, dtype=dt, device=self.device)
                          for _ in range(n_slots)]
        self.compute = torch.cuda.Stream(self.device)
        self.h2d = torch.cuda.Stream(self.device)
        self.d2h = torch.cuda.Stream(self.device)
        self.ev_h2d = [torch.cuda.Event() for _ in range(n_slots)]
        self.ev_comp = [torch.cuda.Event() for _ in range(n_slots)]
        self.ev_d2h = [torch.cuda.Event() for _ in range(n_slots)]
        self.max_tokens = max_tokens
        self.n_submitted = 0

    def submit(self, kv_host: torch.Tensor, emb_host: torch.Tensor, chunk_start, chunk_len,
               out_host: torch.Tensor, inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE):
        """Queue one request: the chunks ``[chunk_start[k], chunk_start[k] + chunk_len[k])``
        of the pinned host pool, in document order.  Returns an event that completes
        when ``out_host[:n_tokens]`` holds the repaired cache (``out_host`` pinned,
        not reused by the caller before then).  Nothing here waits on the GPU."""
        starts = np.asarray(chunk_start, np.int64)
        lens = np.asarray(chunk_len, np.int64)
        n = int(lens.sum())
        if n < 1 or n > self.max_tokens:
            raise ValueError(f"request of {n} tokens: the pipeline holds 1..{self.max_tokens}")
        s = self.n_submitted % self.n_slots
        sess, skv, semb = self.slots[s], self.stage_kv[s], self.stage_emb[s]
        dst = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.int64)
        # this slot's staging pool is free once its previous repair has run
        self.h2d.wait_event(self.ev_comp[s])
        with torch.cuda.stream(self.h2d):
            for a, m, d in zip(starts.tolist(), lens.tolist(), dst.tolist()):
                skv[d:d + m].copy_(kv_host[a:a + m], non_blocking=True)
                semb[d:d + m].copy_(emb_host[a:a + m], non_blocking=True)
            self.ev_h2d[s].record(self.h2d)
        # the chunks have landed, and the slot's previous result has been read back
        self.compute.wait_event(self.ev_h2d[s])
        self.compute.wait_event(self.ev_d2h[s])
        idx = np.arange(len(lens), dtype=np.int32)
        cu = np.array([0, len(lens)], np.int32)
        with torch.cuda.stream(self.compute):
            sess.repair(skv, semb, dst, lens.astype(np.int32), idx, cu, inv_freq_target, rope_mode,
                        stream=self.compute)
            self.ev_comp[s].record(self.compute)
        self.d2h.wait_event(self.ev_comp[s])
        with torch.cuda.stream(self.d2h):
            out_host[:n].copy_(sess.kv[:n], non_blocking=True)
            self.ev_d2h[s].record(self.d2h)
        self.n_submitted += 1
        return self.ev_d2h[s]

    def drain(self):
        """Make the current stream wait for everything submitted so far."""
        cur = torch.cuda.current_stream(self.device)
        for s in range(self.n_slots):
            cur.wait_event(self.ev_d2h[s])


# ------------------------------------------------------------------ training (Sec. 4.2, App. A)
_TRAIN_TOP = ["w_seg", "b_seg", "w_map", "b_map", "w_tok", "b_tok", "w_fuse", "b_fuse", "w_rein", "b_rein"]
_TRAIN_BLOCK = ["ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ln2_g", "ln2_b", "w_fc1", "b_fc1",
                "w_fc2", "b_fc2"]
_TRAIN_END = ["lnf_g", "lnf_b", "w_out", "b_out"]


def trained_tensor_names(n_blocks: int):
    """The trained tensors in the order of the flat parameter vector (include/cr.h)."""
    return _TRAIN_TOP + [f"blk{b}.{k}" for b in range(n_blocks) for k in _TRAIN_BLOCK] + _TRAIN_END


class TrainSession:
    """Training state of the repair network on one GPU: the flat fp32 master weights and
    their bf16 copy, the AdamW moments, the last gradient and the workspace; `step` runs
    one update (forward, objective, backward, clipping, AdamW) through cr_train_step."""

    def __init__(self, target: cr.cr_target_dims, rep: cr.cr_repairer_dims, w: Dict[str, np.ndarray],
                 max_tokens: int, max_request_tokens: int, device="cuda"):
        self.target, self.rep = target, rep
        self.device = torch.device(device)
        self.names = trained_tensor_names(rep.n_blocks)
        self.offsets = cr.cr_param_layout(target, rep)
        P = int(self.offsets[-1])
        flat = np.zeros(P, np.float32)
        for k, name in enumerate(self.names):
            a = np.asarray(w[name])
            a = (a.astype(np.uint32) << 16).view(np.float32) if a.dtype == np.uint16 else a.astype(np.float32)
            flat[self.offsets[k]:self.offsets[k] + a.size] = a.ravel()
        self.params = torch.from_numpy(flat).to(self.device)
        self.params_bf16 = self.params.to(torch.bfloat16)
        self.adam_m = torch.zeros_like(self.params)
        self.adam_v = torch.zeros_like(self.params)
        self.grads = torch.zeros_like(self.params)
        self.sigma_stale = torch.from_numpy(np.asarray(w["sigma_stale"], np.float32)).to(self.device)
        self.sigma_delta = torch.from_numpy(np.asarray(w["sigma_delta"], np.float32)).to(self.device)
        self.stats = torch.zeros(4, dtype=torch.float32, device=self.device)
        ws = cr.cr_train_workspace_bytes(target, rep, max_tokens, max_request_tokens)
        if ws == 0:
            raise cr.CrError("cr_train_workspace_bytes", cr.CR_ERR_INVALID_ARG, "invalid dimensions")
        self.workspace = torch.empty((ws + 15) // 16 * 16, dtype=torch.uint8, device=self.device)
        self.n_steps = 0

    def view(self, t: torch.Tensor, name: str) -> torch.Tensor:
        k = self.names.index(name)
        a, b = int(self.offsets[k]), int(self.offsets[k + 1])
        return t[a:b]

    def step(self, kv_stale, kv_joint, emb, chunk_end, pos, cu_seqlens_host, n_tokens, lr, *,
             beta1=0.9, beta2=0.95, eps=1e-8, weight_decay=0.01, max_grad_norm=1.0, stream=None,
             mask_mode="block_causal"):
        """One AdamW update under mask_mode (the method's mask or an App. F ablation);
        returns the device stats tensor (loss, grad norm, clip coef, 0)."""
        self.n_steps += 1
        hp = cr.cr_adamw(lr, beta1, beta2, eps, weight_decay, max_grad_norm, self.n_steps)
        cr.cr_train_step(self.target, self.rep, self.params, self.params_bf16, self.adam_m, self.adam_v,
                         self.grads, self.sigma_stale, self.sigma_delta, kv_stale, kv_joint, emb, chunk_end,
                         pos, cu_seqlens_host, n_tokens, hp, self.stats, self.workspace, stream,
                         mask_mode)
        return self.stats
