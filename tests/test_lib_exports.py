"""The C-ABI library builds for sm_103a, loads without a GPU, exports every
symbol include/*.h declares, and validates arguments on the host (no device
work is attempted for invalid calls)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_35139_gb300 import build, cr

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return cr.lib()


def _declared():
    names = set()
    for h in ("cr.h", "cr_ops.h"):
        with open(os.path.join(ROOT, "include", h)) as f:
            src = f.read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names |= set(re.findall(r"\b(cr_[a-z0-9_]+)\s*\(", src))
    return sorted(names)


def test_every_declared_symbol_is_exported(L):
    declared = _declared()
    assert len(declared) >= 13
    for name in declared:
        assert hasattr(L, name), name
    assert set(declared) == set(cr.EXPORTED)


def test_library_is_built_for_sm103a_only():
    # the build passes exactly one -gencode for compute_103a / sm_103a
    assert build.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]


def test_status_strings(L):
    for s in range(6):
        assert L.cr_status_str(s)
    assert L.cr_status_str(99) == b"unknown status"


def _dims(name="small"):
    import fixtures as F
    from paper_2609_35139_gb300 import dims_from
    c = F.make_case(name)
    return c, dims_from(c.target, c.repairer)


def test_workspace_bytes_host_logic(L):
    c, (t, r) = _dims("llama8b")
    w1 = cr.cr_workspace_bytes(t, r, 1)
    w2 = cr.cr_workspace_bytes(t, r, 5120)
    assert 0 < w1 < w2
    # dominated by per-token buffers: y (two bf16 terms), s|e (fp32, then two bf16
    # terms), x (fp32), u, qkv, o, g (bf16), the repairer RoPE table (32 (cos, sin)
    # pairs per token), the chunk start (int32) and the pool row (int64)
    per_tok = (2 * 512 * 16 * 2 + 2 * 512 * 4 + 4 * 512 * 2 + 1024 * 4 + 1024 * 2 + 3 * 1024 * 2
               + 1024 * 2 + 4096 * 2 + 32 * 8 + 4 + 8)
    assert abs((w2 - w1) - 5119 * per_tok) < 64 * 256
    bad = cr.repairer_dims(16, 512, 1000, 6, 16, 4096)   # d_b not a multiple of 128
    assert cr.cr_workspace_bytes(t, bad, 10) == 0
    bad = cr.repairer_dims(16, 512, 1024, 6, 8, 4096)    # 128-dim heads: unsupported
    assert cr.cr_workspace_bytes(t, bad, 10) == 0


FAKE = 0x10000   # 16-byte aligned, never dereferenced: validation fails first


def _assemble(L, t, chunk_idx, cu, chunk_len=(10, 20, 30), n_pool=60, max_tokens=1000, ptr=FAKE):
    cs = np.array([0, 10, 30], np.int64)
    cl = np.array(chunk_len, np.int32)
    ci = np.array(chunk_idx, np.int32)
    cc = np.array(cu, np.int32)
    cuh = np.zeros(len(cc), np.int32)
    return L.cr_assemble_stale(ctypes.byref(t), ptr, ptr, n_pool, cs.ctypes.data, cl.ctypes.data,
                               len(cl), ci.ctypes.data, cc.ctypes.data, len(cc) - 1, ptr, ptr,
                               max_tokens, ptr, ptr, ptr, ptr, cuh.ctypes.data, None)


def test_assemble_rejects_bad_inputs_on_host(L):
    c, (t, r) = _dims()
    assert _assemble(L, t, [0, 5], [0, 2]) == cr.CR_ERR_INVALID_ARG        # chunk id out of range
    assert _assemble(L, t, [0, -1], [0, 2]) == cr.CR_ERR_INVALID_ARG
    assert _assemble(L, t, [0, 1], [0, 0, 2]) == cr.CR_ERR_INVALID_ARG     # empty request
    assert _assemble(L, t, [0, 2], [0, 2], n_pool=50) == cr.CR_ERR_INVALID_ARG   # chunk past pool
    assert _assemble(L, t, [0, 1], [0, 2], chunk_len=(10, 0, 30)) == cr.CR_ERR_INVALID_ARG
    assert _assemble(L, t, [2, 1], [0, 2], max_tokens=40) == cr.CR_ERR_INVALID_ARG  # 50 > 40
    assert _assemble(L, t, [0, 1], [0, 2], ptr=FAKE + 8) == cr.CR_ERR_INVALID_ARG  # misaligned
    bad = cr.target_dims(4, 2, 96, 512, "bf16")
    assert _assemble(L, bad, [0, 1], [0, 2]) == cr.CR_ERR_UNSUPPORTED


def test_other_calls_reject_bad_inputs_on_host(L):
    c, (t, r) = _dims()
    w = cr.cr_weights()
    # null weights -> invalid before any device work
    assert L.cr_compress_features(ctypes.byref(t), ctypes.byref(r), ctypes.byref(w), FAKE, FAKE,
                                  10, FAKE, FAKE, FAKE, 1 << 30, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_apply_residual(ctypes.byref(t), ctypes.byref(r), ctypes.byref(w), FAKE, 10, FAKE,
                               FAKE, None, 1, None, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_linear(FAKE, 64, FAKE, None, 10, 30, 64, FAKE, 30, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_linear(FAKE, 64, FAKE, None, 10, 32, 60, FAKE, 32, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_layernorm(FAKE, None, 0, None, FAKE, FAKE, 1e-5, 4, 100, FAKE, None) == \
        cr.CR_ERR_INVALID_ARG
    # cr_matmul: sizes, strides and alignment on the host; widths in 64-column blocks
    assert L.cr_matmul(FAKE, 64, 0, FAKE, 64, 0, 64, 64, FAKE, 64, 0, None, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_matmul(FAKE, 60, 0, FAKE, 64, 10, 64, 60, FAKE, 64, 0, None, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_matmul(FAKE + 8, 64, 0, FAKE, 64, 10, 64, 64, FAKE, 64, 0, None, 0, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_matmul(FAKE, 64, 0, FAKE, 96, 10, 96, 64, FAKE, 96, 0, None, 0, None) == cr.CR_ERR_UNSUPPORTED
    assert L.cr_matmul(FAKE, 96, 1, FAKE, 64, 96, 64, 64, FAKE, 64, 0, None, 0, None) == cr.CR_ERR_UNSUPPORTED
    cu = np.array([0, 100], np.int32)
    assert L.cr_chunk_causal_attention(FAKE, 1024, 8, FAKE, cu.ctypes.data, 1, 100, FAKE,
                                       None) == cr.CR_ERR_UNSUPPORTED          # 128-dim heads
    cu = np.array([0, 100, 90], np.int32)
    assert L.cr_chunk_causal_attention(FAKE, 1024, 16, FAKE, cu.ctypes.data, 2, 90, FAKE,
                                       None) == cr.CR_ERR_INVALID_ARG          # empty request


def test_mask_calls_reject_bad_inputs_on_host(L):
    cu = np.array([0, 100], np.int32)
    att = lambda mode, cend=FAKE, cstart=FAKE, cuv=cu: L.cr_masked_attention(
        FAKE, 512, 8, mode, cend, cstart, cuv.ctypes.data, 1, 100, FAKE, None)
    assert att(7) == cr.CR_ERR_INVALID_ARG                                 # unknown mask
    assert att(-1) == cr.CR_ERR_INVALID_ARG
    assert att(cr.CR_MASK_BLOCK_DIAGONAL, cstart=None) == cr.CR_ERR_INVALID_ARG   # needs starts
    assert att(cr.CR_MASK_BLOCK_CAUSAL, cend=None) == cr.CR_ERR_INVALID_ARG       # needs ends
    assert att(cr.CR_MASK_BLOCK_CAUSAL, cuv=np.array([0, 99], np.int32)) == cr.CR_ERR_INVALID_ARG
    assert L.cr_masked_attention(FAKE, 1024, 8, 1, None, None, cu.ctypes.data, 1, 100, FAKE,
                                 None) == cr.CR_ERR_UNSUPPORTED             # 128-dim heads
    assert L.cr_chunk_starts(FAKE, np.array([0, 99], np.int32).ctypes.data, 1, 100, FAKE,
                             None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_chunk_starts(FAKE + 4, cu.ctypes.data, 1, 100, FAKE, None) == cr.CR_ERR_INVALID_ARG
    c, (t, r) = _dims()
    w = cr.cr_weights()
    w.lnf_g = w.lnf_b = FAKE
    assert L.cr_repair_forward_masked(ctypes.byref(t), ctypes.byref(r), ctypes.byref(w), FAKE, FAKE,
                                      FAKE, FAKE, cu.ctypes.data, 1, 100, 9, FAKE, FAKE, 1 << 30,
                                      None) == cr.CR_ERR_INVALID_ARG


def test_output_choice_calls_reject_bad_inputs_on_host(L):
    c, (t, r) = _dims()
    w = cr.cr_weights()
    w.w_out = w.b_out = w.sigma_delta = FAKE
    sel = lambda tt, comp=3, off=0, keep=None, rope=0, freq=None: L.cr_apply_residual_select(
        ctypes.byref(tt), ctypes.byref(r), ctypes.byref(w), FAKE, 10, FAKE, FAKE, freq, rope, comp,
        off, keep, None, 0, None)
    for comp in (0, 4, -1):
        assert sel(t, comp=comp) == cr.CR_ERR_INVALID_ARG
    assert sel(t, off=2) == cr.CR_ERR_INVALID_ARG
    assert sel(t, keep=FAKE + 4) == cr.CR_ERR_INVALID_ARG                 # misaligned chunk map
    assert sel(t, rope=cr.CR_ROPE_GLOBAL) == cr.CR_ERR_INVALID_ARG         # R_M needs frequencies
    one_head = cr.target_dims(4, 1, 128, 512, "bf16")                      # H d_h = 128 < 256
    assert sel(one_head, comp=cr.CR_APPLY_K) == cr.CR_ERR_UNSUPPORTED
    f = np.ones(64, np.float32)
    assert L.cr_rotate_k(ctypes.byref(t), FAKE, 10, FAKE, None, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_rotate_k(ctypes.byref(t), FAKE + 8, 10, FAKE, f.ctypes.data, None) == cr.CR_ERR_INVALID_ARG
    assert L.cr_rotate_k(ctypes.byref(t), FAKE, 0, FAKE, f.ctypes.data, None) == cr.CR_ERR_INVALID_ARG


def test_paged_residual_rejects_bad_inputs_on_host(L):
    c, (t, r) = _dims()
    w = cr.cr_weights()
    w.w_out = w.b_out = w.sigma_delta = FAKE
    call = lambda tt, n=10, slots=64, paged=FAKE: L.cr_apply_residual_paged(
        ctypes.byref(tt), ctypes.byref(r), ctypes.byref(w), FAKE, n, FAKE, FAKE, None, 0, FAKE, paged,
        slots, None, 0, None)
    assert call(t, slots=0) == cr.CR_ERR_INVALID_ARG          # no slots
    assert call(t, n=0) == cr.CR_ERR_INVALID_ARG              # no tokens
    assert call(t, paged=FAKE + 8) == cr.CR_ERR_INVALID_ARG   # misaligned cache
    f32 = cr.target_dims(4, 2, 128, 512, "f32")
    assert call(f32) == cr.CR_ERR_UNSUPPORTED                 # bf16 caches only
    narrow = cr.target_dims(4, 1, 128, 512, "bf16")           # H_kv d_h = 128: not a multiple of 256
    assert call(narrow) == cr.CR_ERR_UNSUPPORTED


def test_fused_front_rejects_bad_inputs_on_host(L):
    """cr_assemble_compress checks the chunk map, weights and workspace before any launch."""
    c, (t, r) = _dims()
    w = cr.cr_weights()
    for f in ("w_seg", "b_seg", "w_map", "b_map", "w_tok", "b_tok", "w_fuse", "b_fuse", "w_rein",
              "b_rein", "sigma_stale"):
        setattr(w, f, FAKE)
    ws = cr.cr_workspace_bytes(t, r, 1000)

    def call(chunk_idx, cu, chunk_len=(10, 20, 30), n_pool=60, max_tokens=1000, ptr=FAKE,
             weights=w, ws_bytes=ws):
        cs = np.array([0, 10, 30], np.int64)
        cl = np.array(chunk_len, np.int32)
        ci = np.array(chunk_idx, np.int32)
        cc = np.array(cu, np.int32)
        cuh = np.zeros(len(cc), np.int32)
        return L.cr_assemble_compress(ctypes.byref(t), ctypes.byref(r), ctypes.byref(weights), ptr,
                                      ptr, n_pool, cs.ctypes.data, cl.ctypes.data, len(cl),
                                      ci.ctypes.data, cc.ctypes.data, len(cc) - 1, ptr, ptr,
                                      max_tokens, ptr, ptr, ptr, ptr, cuh.ctypes.data, FAKE, FAKE,
                                      FAKE, ws_bytes, None)

    assert call([0, 5], [0, 2]) == cr.CR_ERR_INVALID_ARG          # chunk id out of range
    assert call([0, 1], [0, 0, 2]) == cr.CR_ERR_INVALID_ARG       # empty request
    assert call([0, 2], [0, 2], n_pool=50) == cr.CR_ERR_INVALID_ARG   # chunk past the pool
    assert call([0, 1], [0, 2], chunk_len=(10, 0, 30)) == cr.CR_ERR_INVALID_ARG
    assert call([2, 1], [0, 2], max_tokens=40) == cr.CR_ERR_INVALID_ARG
    assert call([0, 1], [0, 2], ptr=FAKE + 8) == cr.CR_ERR_INVALID_ARG   # misaligned
    assert call([0, 1], [0, 2], weights=cr.cr_weights()) == cr.CR_ERR_INVALID_ARG   # no weights
    assert call([0, 1], [0, 2], ws_bytes=ws - 256) == cr.CR_ERR_INVALID_ARG    # workspace short
    bad = cr.repairer_dims(12, 128, 256, 2, 4, 1024)    # d_seg 12: unsupported
    assert L.cr_assemble_compress(ctypes.byref(t), ctypes.byref(bad), ctypes.byref(w), *([FAKE] * 2),
                                  60, None, None, 3, None, None, 1, *([FAKE] * 2), 100,
                                  *([FAKE] * 4), None, FAKE, FAKE, FAKE, ws, None) == \
        cr.CR_ERR_UNSUPPORTED


def test_pool_head_rejects_bad_inputs_on_host(L):
    """cr_apply_residual_pool checks its dims, pointers, RoPE mode and workspace before
    it reads the chunk map or launches anything."""
    c, (t, r) = _dims()
    w = cr.cr_weights()
    w.w_out = w.b_out = w.sigma_delta = FAKE
    ws = cr.cr_workspace_bytes(t, r, 100)
    freq = np.ones(64, np.float32)

    def call(tt=t, n=100, n_pool=60, yf=FAKE, kv_pool=FAKE, kv_out=FAKE, rope=cr.CR_ROPE_NONE,
             inv_freq=None, workspace=FAKE, ws_bytes=ws, weights=w):
        return L.cr_apply_residual_pool(ctypes.byref(tt), ctypes.byref(r), ctypes.byref(weights), yf, n,
                                        kv_pool, n_pool, None, None, 3, None, None, 1, kv_out, FAKE,
                                        inv_freq, rope, workspace, ws_bytes, None)

    assert call(tt=cr.target_dims(4, 2, 128, 512, "f32")) == cr.CR_ERR_UNSUPPORTED   # bf16 caches only
    assert call(n=0) == cr.CR_ERR_INVALID_ARG                      # no tokens
    assert call(n_pool=0) == cr.CR_ERR_INVALID_ARG                 # empty pool
    assert call(kv_pool=None) == cr.CR_ERR_INVALID_ARG             # no pool
    assert call(kv_out=None) == cr.CR_ERR_INVALID_ARG              # no output
    assert call(workspace=None) == cr.CR_ERR_INVALID_ARG           # no workspace
    assert call(yf=FAKE + 8) == cr.CR_ERR_INVALID_ARG              # misaligned
    assert call(rope=7) == cr.CR_ERR_INVALID_ARG                   # unknown RoPE mode
    assert call(rope=cr.CR_ROPE_GLOBAL) == cr.CR_ERR_INVALID_ARG   # R_M without frequencies
    assert call(ws_bytes=ws - 256) == cr.CR_ERR_INVALID_ARG        # workspace short
    assert call(weights=cr.cr_weights()) == cr.CR_ERR_INVALID_ARG  # no head weights
    odd = cr.target_dims(3, 1, 64, 512, "bf16")                    # D_KV = 384: not whole 256-column tiles
    assert call(tt=odd, inv_freq=freq.ctypes.data) == cr.CR_ERR_UNSUPPORTED
