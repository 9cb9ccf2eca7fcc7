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
        self.rein = z(n, max(rep.n_blocks, 1) * rep.d_b, dtype=torch.bfloat16)
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

    def forward(self, a: Assembled, stream=None):
        cr.cr_repair_forward(self.target, self.rep, self.weights, self.h0, self.rein,
                             self.chunk_end, self.pos, a.cu_seqlens, a.n_tokens, self.yf,
                             self.workspace, stream)

    def apply(self, a: Assembled, inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None):
        cr.cr_apply_residual(self.target, self.rep, self.weights, self.yf, a.n_tokens, self.kv,
                             self.pos, inv_freq_target, rope_mode, stream)

    def repair(self, kv_pool, emb_pool, chunk_start, chunk_len, chunk_idx, cu_chunks,
               inv_freq_target=None, rope_mode=cr.CR_ROPE_NONE, stream=None) -> Assembled:
        """Assemble, compress, run the blocks and apply the residual; kv holds the result."""
        a = self.assemble(kv_pool, emb_pool, chunk_start, chunk_len, chunk_idx, cu_chunks, stream)
        self.compress(a, stream)
        self.forward(a, stream)
        self.apply(a, inv_freq_target, rope_mode, stream)
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
