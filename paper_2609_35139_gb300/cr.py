"""ctypes binding of the repair library's C ABI (include/cr.h, include/cr_ops.h).

Argument marshalling only: every function here forwards torch tensors' device
pointers, host arrays and the current CUDA stream to the function of the same
name in libcacherepair.so.  There is no fallback: if the library is not built
or a call fails, a CrError is raised.
"""
from __future__ import annotations

import ctypes
import os
from ctypes import POINTER, c_float, c_int32, c_int64, c_size_t, c_uint32, c_void_p
from typing import Dict, Optional, Sequence

import numpy as np
import torch

from . import build as _build

CR_OK, CR_ERR_INVALID_ARG, CR_ERR_UNSUPPORTED, CR_ERR_CUDA, CR_ERR_DEVICE_INDEX, CR_ERR_TIMEOUT = range(6)
CR_F32, CR_BF16 = 0, 1
CR_ROPE_NONE, CR_ROPE_GLOBAL = 0, 1
CR_EPI_BF16, CR_EPI_GELU_BF16, CR_EPI_ADD_F32, CR_EPI_F32 = range(4)

EXPORTED = [
    "cr_workspace_bytes", "cr_assemble_stale", "cr_compress_features", "cr_assemble_compress",
    "cr_repair_forward",
    "cr_repair_forward_masked", "cr_apply_residual", "cr_apply_residual_select", "cr_rotate_k",
    "cr_apply_residual_paged", "cr_apply_residual_pool", "cr_canonicalize_chunks",
    "cr_sigma_workspace_bytes", "cr_sigma_accumulate", "cr_sigma_finalize", "cr_get_device_status",
    "cr_clear_device_status", "cr_status_str", "cr_last_cuda_error",
    "cr_linear", "cr_matmul", "cr_layernorm", "cr_chunk_causal_attention", "cr_masked_attention",
    "cr_chunk_starts", "cr_qkv_rope", "cr_segment_project",
    "cr_segment_project_noalloc", "cr_param_layout", "cr_train_workspace_bytes", "cr_train_step",
    "cr_wait_selftest",
]


class CrError(RuntimeError):
    def __init__(self, name: str, status: int, text: str):
        super().__init__(f"{name} failed: {text} (status {status})")
        self.status = status


class cr_target_dims(ctypes.Structure):
    _fields_ = [("n_layers", c_int32), ("n_kv_heads", c_int32), ("head_dim", c_int32),
                ("d_model", c_int32), ("cache_dtype", c_int32)]


class cr_repairer_dims(ctypes.Structure):
    _fields_ = [("d_seg", c_int32), ("d_c", c_int32), ("d_b", c_int32), ("n_blocks", c_int32),
                ("n_heads", c_int32), ("mlp_hidden", c_int32), ("ln_eps", c_float),
                ("rope_theta", c_float)]


_BLOCK_FIELDS = ["ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ln2_g", "ln2_b", "w_fc1",
                 "b_fc1", "w_fc2", "b_fc2"]
_WEIGHT_FIELDS = ["w_seg", "b_seg", "w_map", "b_map", "w_tok", "b_tok", "w_fuse", "b_fuse",
                  "w_rein", "b_rein", "blocks", "lnf_g", "lnf_b", "w_out", "b_out",
                  "sigma_stale", "sigma_delta"]


class cr_block_weights(ctypes.Structure):
    _fields_ = [(f, c_void_p) for f in _BLOCK_FIELDS]


class cr_weights(ctypes.Structure):
    _fields_ = [(f, c_void_p) for f in _WEIGHT_FIELDS]


class cr_adamw(ctypes.Structure):
    _fields_ = [("lr", c_float), ("beta1", c_float), ("beta2", c_float), ("eps", c_float),
                ("weight_decay", c_float), ("max_grad_norm", c_float), ("step", c_int32)]


_lib_handle = None


def lib(build_if_missing: bool = False) -> ctypes.CDLL:
    """Load libcacherepair.so (raises if it is absent, unless asked to build it)."""
    global _lib_handle
    if _lib_handle is not None:
        return _lib_handle
    path = _build.LIB_PATH
    if build_if_missing:
        path = _build.build()
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is not built; run paper_2609_35139_gb300.build.build() "
                           "(or __graft_entry__.build()) first")
    L = ctypes.CDLL(path)
    vp, i32, i64 = c_void_p, c_int32, c_int64
    P = ctypes.POINTER
    sig = {
        "cr_workspace_bytes": (c_size_t, [P(cr_target_dims), P(cr_repairer_dims), i64]),
        "cr_assemble_stale": (i32, [P(cr_target_dims), vp, vp, i64, vp, vp, i32, vp, vp, i32, vp,
                                    vp, i64, vp, vp, vp, vp, vp, vp]),
        "cr_compress_features": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp,
                                       vp, i64, vp, vp, vp, c_size_t, vp]),
        "cr_assemble_compress": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp,
                                       vp, i64, vp, vp, i32, vp, vp, i32, vp, vp, i64, vp, vp, vp,
                                       vp, vp, vp, vp, vp, c_size_t, vp]),
        "cr_repair_forward": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp, vp,
                                    vp, vp, vp, i32, i64, vp, vp, c_size_t, vp]),
        "cr_repair_forward_masked": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights),
                                           vp, vp, vp, vp, vp, i32, i64, i32, vp, vp, c_size_t,
                                           vp]),
        "cr_apply_residual": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp, i64,
                                    vp, vp, vp, i32, vp, c_size_t, vp]),
        "cr_apply_residual_paged": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp,
                                          i64, vp, vp, vp, i32, vp, vp, i64, vp, c_size_t, vp]),
        "cr_apply_residual_pool": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp, i64,
                                         vp, i64, vp, vp, i32, vp, vp, i32, vp, vp, vp, i32, vp, c_size_t,
                                         vp]),
        "cr_canonicalize_chunks": (i32, [P(cr_target_dims), vp, i64, vp, vp, vp]),
        "cr_rotate_k": (i32, [P(cr_target_dims), vp, i64, vp, vp, vp]),
        "cr_apply_residual_select": (i32, [P(cr_target_dims), P(cr_repairer_dims), P(cr_weights), vp,
                                           i64, vp, vp, vp, i32, i32, i32, vp, vp, c_size_t, vp]),
        "cr_sigma_workspace_bytes": (ctypes.c_size_t, [P(cr_target_dims), i64]),
        "cr_sigma_accumulate": (i32, [P(cr_target_dims), vp, vp, i64, vp, vp, ctypes.c_size_t, vp]),
        "cr_sigma_finalize": (i32, [P(cr_target_dims), vp, i64, vp, vp]),
        "cr_get_device_status": (i32, [P(c_uint32)]),
        "cr_clear_device_status": (i32, []),
        "cr_status_str": (ctypes.c_char_p, [i32]),
        "cr_last_cuda_error": (ctypes.c_char_p, []),
        "cr_linear": (i32, [vp, i64, vp, vp, i64, i64, i64, vp, i64, i32, vp]),
        "cr_matmul": (i32, [vp, i64, i32, vp, i64, i64, i64, i64, vp, i64, i32, vp, c_size_t, vp]),
        "cr_layernorm": (i32, [vp, vp, i64, vp, vp, vp, c_float, i64, i64, vp, vp]),
        "cr_chunk_causal_attention": (i32, [vp, i32, i32, vp, vp, i32, i64, vp, vp]),
        "cr_param_layout": (i32, [P(cr_target_dims), P(cr_repairer_dims), vp, i32]),
        "cr_wait_selftest": (i32, [vp]),
        "cr_train_workspace_bytes": (c_size_t, [P(cr_target_dims), P(cr_repairer_dims), i64, i64]),
        "cr_train_step": (i32, [P(cr_target_dims), P(cr_repairer_dims), vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                vp, vp, vp, vp, i32, i64, i32, P(cr_adamw), vp, vp, c_size_t, vp]),
        "cr_masked_attention": (i32, [vp, i32, i32, i32, vp, vp, vp, i32, i64, vp, vp]),
        "cr_chunk_starts": (i32, [vp, vp, i32, i64, vp, vp]),
        "cr_qkv_rope": (i32, [vp, vp, vp, vp, i64, i32, i32, c_float, vp, vp]),
        "cr_segment_project": (i32, [P(cr_target_dims), i32, vp, i64, vp, vp, vp, vp, vp, c_size_t,
                                     vp]),
        "cr_segment_project_noalloc": (i32, [P(cr_target_dims), i32, vp, i64, vp, vp, vp, vp, vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib_handle = L
    return L


def _check(name: str, status: int):
    if status != CR_OK:
        text = lib().cr_status_str(status).decode()
        if status == CR_ERR_CUDA:
            text += ": " + lib().cr_last_cuda_error().decode()
        raise CrError(name, status, text)


def _p(t) -> Optional[int]:
    """Device pointer of a tensor (None -> NULL)."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else stream


def _host_arr(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a), dtype=dtype)


def target_dims(n_layers, n_kv_heads, head_dim, d_model, cache_dtype) -> cr_target_dims:
    dt = cache_dtype if isinstance(cache_dtype, int) else (CR_F32 if cache_dtype == "f32" else CR_BF16)
    return cr_target_dims(n_layers, n_kv_heads, head_dim, d_model, dt)


def repairer_dims(d_seg, d_c, d_b, n_blocks, n_heads, mlp_hidden, ln_eps=1e-5,
                  rope_theta=1e4) -> cr_repairer_dims:
    return cr_repairer_dims(d_seg, d_c, d_b, n_blocks, n_heads, mlp_hidden, ln_eps, rope_theta)


class PackedWeights:
    """cr_weights for a dict of device tensors (keeps the tensors and the block array alive).

    Keys follow cr.h: w_seg, b_seg, ..., w_out, b_out, sigma_stale, sigma_delta, and
    per block ``blk{b}.<field>``.  Stacked reinjection weights (w_rein [B, d_b, d_c],
    b_rein [B, d_b]) are passed as one [B d_b, d_c] matrix, as the header states.
    """

    def __init__(self, tensors: Dict[str, torch.Tensor], n_blocks: int):
        self.tensors = tensors
        self.blocks = (cr_block_weights * max(n_blocks, 1))()
        for b in range(n_blocks):
            for f in _BLOCK_FIELDS:
                setattr(self.blocks[b], f, _p(tensors[f"blk{b}.{f}"]))
        self.struct = cr_weights()
        for f in _WEIGHT_FIELDS:
            if f == "blocks":
                self.struct.blocks = ctypes.cast(self.blocks, c_void_p)
            else:
                t = tensors.get(f)
                setattr(self.struct, f, _p(t) if t is not None else None)


# ------------------------------------------------------------------ cr.h
def cr_workspace_bytes(target: cr_target_dims, rep: cr_repairer_dims, max_tokens: int) -> int:
    return int(lib().cr_workspace_bytes(ctypes.byref(target), ctypes.byref(rep), max_tokens))


def cr_assemble_stale(target, kv_pool, emb_pool, chunk_start, chunk_len, chunk_idx, cu_chunks,
                      kv_out, emb_out, chunk_id, chunk_end, pos, cu_seqlens_dev, stream=None):
    """Returns (n_tokens, cu_seqlens_host int32 array)."""
    cs = _host_arr(chunk_start, np.int64)
    cl = _host_arr(chunk_len, np.int32)
    ci = _host_arr(chunk_idx, np.int32)
    cu = _host_arr(cu_chunks, np.int32)
    n_req = len(cu) - 1
    cu_host = np.zeros(max(n_req + 1, 1), np.int32)
    n_pool = kv_pool.shape[0]
    st = lib().cr_assemble_stale(
        ctypes.byref(target), _p(kv_pool), _p(emb_pool), n_pool, cs.ctypes.data, cl.ctypes.data,
        len(cl), ci.ctypes.data, cu.ctypes.data, n_req, _p(kv_out), _p(emb_out), kv_out.shape[0],
        _p(chunk_id), _p(chunk_end), _p(pos), _p(cu_seqlens_dev), cu_host.ctypes.data,
        _stream(stream))
    _check("cr_assemble_stale", st)
    return int(cu_host[-1]), cu_host


def cr_compress_features(target, rep, weights: PackedWeights, kv, emb, n_tokens, h0_out,
                         rein_out, workspace, stream=None):
    st = lib().cr_compress_features(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(kv), _p(emb),
        n_tokens, _p(h0_out), _p(rein_out), _p(workspace), workspace.numel() * workspace.element_size(),
        _stream(stream))
    _check("cr_compress_features", st)


def cr_assemble_compress(target, rep, weights: PackedWeights, kv_pool, emb_pool, chunk_start,
                         chunk_len, chunk_idx, cu_chunks, kv_out, emb_out, chunk_id, chunk_end, pos,
                         cu_seqlens_dev, h0_out, rein_out, workspace, stream=None):
    """cr_assemble_stale + cr_compress_features in one call; returns (n_tokens, cu_seqlens_host).
    kv_out None (bf16 caches): the assembled cache is not written (see cr_apply_residual_pool)."""
    cs = _host_arr(chunk_start, np.int64)
    cl = _host_arr(chunk_len, np.int32)
    ci = _host_arr(chunk_idx, np.int32)
    cu = _host_arr(cu_chunks, np.int32)
    n_req = len(cu) - 1
    cu_host = np.zeros(max(n_req + 1, 1), np.int32)
    st = lib().cr_assemble_compress(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(kv_pool),
        _p(emb_pool), kv_pool.shape[0], cs.ctypes.data, cl.ctypes.data, len(cl), ci.ctypes.data,
        cu.ctypes.data, n_req, _p(kv_out), _p(emb_out), emb_out.shape[0], _p(chunk_id),
        _p(chunk_end), _p(pos), _p(cu_seqlens_dev), cu_host.ctypes.data, _p(h0_out), _p(rein_out),
        _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream))
    _check("cr_assemble_compress", st)
    return int(cu_host[-1]), cu_host


def cr_repair_forward(target, rep, weights: PackedWeights, h0, rein, chunk_end, pos,
                      cu_seqlens_host, n_tokens, yf_out, workspace, stream=None):
    cu = _host_arr(cu_seqlens_host, np.int32)
    st = lib().cr_repair_forward(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(h0), _p(rein),
        _p(chunk_end), _p(pos), cu.ctypes.data, len(cu) - 1, n_tokens, _p(yf_out), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream))
    _check("cr_repair_forward", st)


CR_MASK_BLOCK_CAUSAL, CR_MASK_TOKEN_CAUSAL, CR_MASK_BIDIRECTIONAL, CR_MASK_BLOCK_DIAGONAL = 0, 1, 2, 3
MASK_MODES = {"block_causal": CR_MASK_BLOCK_CAUSAL, "token_causal": CR_MASK_TOKEN_CAUSAL,
              "bidirectional": CR_MASK_BIDIRECTIONAL, "block_diagonal": CR_MASK_BLOCK_DIAGONAL}


def _mask_mode(mode):
    return MASK_MODES[mode] if isinstance(mode, str) else int(mode)


def cr_repair_forward_masked(target, rep, weights: PackedWeights, h0, rein, chunk_end, pos,
                             cu_seqlens_host, n_tokens, mask_mode, yf_out, workspace, stream=None):
    cu = _host_arr(cu_seqlens_host, np.int32)
    st = lib().cr_repair_forward_masked(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(h0), _p(rein),
        _p(chunk_end), _p(pos), cu.ctypes.data, len(cu) - 1, n_tokens, _mask_mode(mask_mode),
        _p(yf_out), _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream))
    _check("cr_repair_forward_masked", st)


def _ws(workspace):
    return (None, 0) if workspace is None else (_p(workspace), workspace.numel() * workspace.element_size())


def cr_apply_residual(target, rep, weights: PackedWeights, yf, n_tokens, kv_inout, pos,
                      inv_freq_host=None, rope_mode=CR_ROPE_NONE, workspace=None, stream=None):
    f = None if inv_freq_host is None else _host_arr(inv_freq_host, np.float32)
    st = lib().cr_apply_residual(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(yf), n_tokens,
        _p(kv_inout), _p(pos), None if f is None else f.ctypes.data, rope_mode, *_ws(workspace),
        _stream(stream))
    _check("cr_apply_residual", st)


def cr_apply_residual_pool(target, rep, weights: PackedWeights, yf, n_tokens, kv_pool, chunk_start,
                           chunk_len, chunk_idx, cu_chunks, kv_out, pos, inv_freq_host=None,
                           rope_mode=CR_ROPE_NONE, workspace=None, stream=None):
    """The head with the stale rows read from the pool, the repaired rows written to kv_out."""
    cs = _host_arr(chunk_start, np.int64)
    cl = _host_arr(chunk_len, np.int32)
    ci = _host_arr(chunk_idx, np.int32)
    cu = _host_arr(cu_chunks, np.int32)
    f = None if inv_freq_host is None else _host_arr(inv_freq_host, np.float32)
    st = lib().cr_apply_residual_pool(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(yf), n_tokens,
        _p(kv_pool), kv_pool.shape[0], cs.ctypes.data, cl.ctypes.data, len(cl), ci.ctypes.data,
        cu.ctypes.data, len(cu) - 1, _p(kv_out), _p(pos), None if f is None else f.ctypes.data,
        rope_mode, *_ws(workspace), _stream(stream))
    _check("cr_apply_residual_pool", st)


CR_APPLY_K, CR_APPLY_V, CR_APPLY_KV = 1, 2, 3
CR_OFFSET_STALE, CR_OFFSET_ZERO = 0, 1
COMPONENTS = {"k": CR_APPLY_K, "v": CR_APPLY_V, "kv": CR_APPLY_KV}
OFFSETS = {"stale": CR_OFFSET_STALE, "zero": CR_OFFSET_ZERO}


def cr_apply_residual_select(target, rep, weights: PackedWeights, yf, n_tokens, kv_inout, pos,
                             inv_freq_host=None, rope_mode=CR_ROPE_NONE, component="kv",
                             offset="stale", keep_chunk_id=None, workspace=None, stream=None):
    """Head + residual add under an output choice (K only / V only, zero offset,
    first chunk kept stale when keep_chunk_id is the chunk map)."""
    f = None if inv_freq_host is None else _host_arr(inv_freq_host, np.float32)
    comp = COMPONENTS[component] if isinstance(component, str) else int(component)
    off = OFFSETS[offset] if isinstance(offset, str) else int(offset)
    st = lib().cr_apply_residual_select(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(yf), n_tokens,
        _p(kv_inout), _p(pos), None if f is None else f.ctypes.data, rope_mode, comp, off,
        _p(keep_chunk_id), *_ws(workspace), _stream(stream))
    _check("cr_apply_residual_select", st)


def cr_rotate_k(target, kv_inout, n_tokens, pos, inv_freq_host, stream=None):
    """K <- R_M(pos) K in place (the stale cache's re-rotation of canonical K)."""
    f = _host_arr(inv_freq_host, np.float32)
    _check("cr_rotate_k", lib().cr_rotate_k(
        ctypes.byref(target), _p(kv_inout), n_tokens, _p(pos), f.ctypes.data, _stream(stream)))


def cr_apply_residual_paged(target, rep, weights: PackedWeights, yf, n_tokens, kv_stale, pos,
                            slot_mapping, paged_cache, num_slots, inv_freq_host=None,
                            rope_mode=CR_ROPE_NONE, workspace=None, stream=None):
    """Head + residual add, repaired rows written to paged_cache[(2l+kv)*num_slots + slot]."""
    f = None if inv_freq_host is None else _host_arr(inv_freq_host, np.float32)
    st = lib().cr_apply_residual_paged(
        ctypes.byref(target), ctypes.byref(rep), ctypes.byref(weights.struct), _p(yf), n_tokens,
        _p(kv_stale), _p(pos), None if f is None else f.ctypes.data, rope_mode, _p(slot_mapping),
        _p(paged_cache), num_slots, *_ws(workspace), _stream(stream))
    _check("cr_apply_residual_paged", st)


def cr_canonicalize_chunks(target, kv_inout, n_tokens, pos, inv_freq_host, stream=None):
    f = _host_arr(inv_freq_host, np.float32)
    _check("cr_canonicalize_chunks", lib().cr_canonicalize_chunks(
        ctypes.byref(target), _p(kv_inout), n_tokens, _p(pos), f.ctypes.data, _stream(stream)))


def cr_sigma_workspace_bytes(target, n_tokens) -> int:
    return int(lib().cr_sigma_workspace_bytes(ctypes.byref(target), n_tokens))


def cr_sigma_accumulate(target, a, b, n_tokens, sumsq, workspace, stream=None):
    _check("cr_sigma_accumulate", lib().cr_sigma_accumulate(
        ctypes.byref(target), _p(a), _p(b), n_tokens, _p(sumsq), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def cr_sigma_finalize(target, sumsq, count, sigma_out, stream=None):
    _check("cr_sigma_finalize", lib().cr_sigma_finalize(
        ctypes.byref(target), _p(sumsq), count, _p(sigma_out), _stream(stream)))


def cr_get_device_status():
    out = (c_uint32 * 3)()
    st = lib().cr_get_device_status(out)
    return st, list(out)


def cr_clear_device_status():
    _check("cr_clear_device_status", lib().cr_clear_device_status())


# ------------------------------------------------------------------ cr_ops.h
def cr_linear(A, W, bias, out, epi=CR_EPI_BF16, M=None, N=None, K=None, lda=None, ldo=None,
              stream=None):
    M = A.shape[0] if M is None else M
    K = W.shape[1] if K is None else K
    N = W.shape[0] if N is None else N
    lda = A.stride(0) if lda is None else lda
    ldo = out.stride(0) if ldo is None else ldo
    _check("cr_linear", lib().cr_linear(_p(A), lda, _p(W), _p(bias), M, N, K, _p(out), ldo, epi,
                                        _stream(stream)))


def cr_matmul(A, B, C, a_trans=False, accumulate=False, workspace=None, stream=None):
    """C [M, N] fp32 (+)= op(A) B; B [K, N] bf16; op(A) = A [M, K] or, with a_trans, A.T for A [K, M].
    An optional workspace lets the product run as k-parts summed in a fixed order."""
    K, N = B.shape
    M = A.shape[1] if a_trans else A.shape[0]
    _check("cr_matmul", lib().cr_matmul(_p(A), A.stride(0), int(bool(a_trans)), _p(B), B.stride(0), M, N, K,
                                        _p(C), C.stride(0), int(bool(accumulate)), *_ws(workspace),
                                        _stream(stream)))


def cr_layernorm(x, gamma, beta, eps, u, add=None, ld_add=0, x_out=None, stream=None):
    M, D = x.shape
    _check("cr_layernorm", lib().cr_layernorm(_p(x), _p(add), ld_add, _p(x_out), _p(gamma),
                                              _p(beta), eps, M, D, _p(u), _stream(stream)))


def cr_chunk_causal_attention(qkv, d_b, n_heads, chunk_end, cu_seqlens_host, out, stream=None):
    cu = _host_arr(cu_seqlens_host, np.int32)
    _check("cr_chunk_causal_attention", lib().cr_chunk_causal_attention(
        _p(qkv), d_b, n_heads, _p(chunk_end), cu.ctypes.data, len(cu) - 1, qkv.shape[0], _p(out),
        _stream(stream)))


def cr_wait_selftest(stream=None):
    """Launch the bounded-wait check (a wait that must time out and report it)."""
    _check("cr_wait_selftest", lib().cr_wait_selftest(_stream(stream)))


def cr_param_layout(target, rep) -> np.ndarray:
    """Offsets of the trained tensors in the flat parameter vector (last entry: the total)."""
    off = np.zeros(14 + 12 * 64 + 1, np.int64)
    _check("cr_param_layout", lib().cr_param_layout(ctypes.byref(target), ctypes.byref(rep),
                                                    off.ctypes.data, len(off)))
    return off[:14 + 12 * rep.n_blocks + 1].copy()


def cr_train_workspace_bytes(target, rep, max_tokens, max_request_tokens) -> int:
    return int(lib().cr_train_workspace_bytes(ctypes.byref(target), ctypes.byref(rep), max_tokens,
                                              max_request_tokens))


def cr_train_step(target, rep, params, params_bf16, adam_m, adam_v, grads, sigma_stale, sigma_delta,
                  kv_stale, kv_joint, emb, chunk_end, pos, cu_seqlens_host, n_tokens, hp: "cr_adamw",
                  stats_out, workspace, stream=None, mask_mode="block_causal"):
    cu = _host_arr(cu_seqlens_host, np.int32)
    _check("cr_train_step", lib().cr_train_step(
        ctypes.byref(target), ctypes.byref(rep), _p(params), _p(params_bf16), _p(adam_m), _p(adam_v),
        _p(grads), _p(sigma_stale), _p(sigma_delta), _p(kv_stale), _p(kv_joint), _p(emb), _p(chunk_end),
        _p(pos), cu.ctypes.data, len(cu) - 1, n_tokens, _mask_mode(mask_mode), ctypes.byref(hp),
        _p(stats_out), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def cr_masked_attention(qkv, d_b, n_heads, mask_mode, chunk_end, chunk_start, cu_seqlens_host, out,
                        stream=None):
    cu = _host_arr(cu_seqlens_host, np.int32)
    _check("cr_masked_attention", lib().cr_masked_attention(
        _p(qkv), d_b, n_heads, _mask_mode(mask_mode), _p(chunk_end), _p(chunk_start), cu.ctypes.data,
        len(cu) - 1, qkv.shape[0], _p(out), _stream(stream)))


def cr_chunk_starts(chunk_end, cu_seqlens_host, n_tokens, chunk_start, stream=None):
    cu = _host_arr(cu_seqlens_host, np.int32)
    _check("cr_chunk_starts", lib().cr_chunk_starts(
        _p(chunk_end), cu.ctypes.data, len(cu) - 1, n_tokens, _p(chunk_start), _stream(stream)))


def cr_qkv_rope(u, w_qkv, b_qkv, pos, d_b, n_heads, rope_theta, qkv, stream=None):
    _check("cr_qkv_rope", lib().cr_qkv_rope(_p(u), _p(w_qkv), _p(b_qkv), _p(pos), u.shape[0], d_b,
                                            n_heads, rope_theta, _p(qkv), _stream(stream)))


def cr_segment_project(target, d_seg, kv, w_seg, b_seg, sigma_stale, y, workspace, stream=None):
    _check("cr_segment_project", lib().cr_segment_project(
        ctypes.byref(target), d_seg, _p(kv), kv.shape[0], _p(w_seg), _p(b_seg), _p(sigma_stale),
        _p(y), _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


def cr_segment_project_noalloc(target, d_seg, kv, w_seg, b_seg, sigma_stale, y, stream=None):
    """cr_segment_project for callers that cannot allocate: no workspace argument."""
    _check("cr_segment_project_noalloc", lib().cr_segment_project_noalloc(
        ctypes.byref(target), d_seg, _p(kv), kv.shape[0], _p(w_seg), _p(b_seg), _p(sigma_stale),
        _p(y), _stream(stream)))
