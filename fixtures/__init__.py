"""Seeded synthetic inputs for the repair path: caches, embeddings, chunk maps, weights, sigma.

This module is the only code shared by the test oracle and the GPU path.  It
holds none of the repair method's arithmetic: it draws numbers (``gen.c``,
counter-based SplitMix64 + Box-Muller) and lays them out in the shapes of the
paper's workloads.  Nothing here reads a dataset; every value is synthetic.

Layout conventions (the same ones the library's C header documents):
  * cache rows are token-major: ``kv[t, j]`` with
    ``j = ((layer * 2 + kv) * n_kv_heads + head) * head_dim + d``, kv = 0 for K
    (canonical, un-rotated K, Section 4.1 "Chunk-cache preparation");
  * a pool holds independently prefilled chunks back to back; chunk ``c`` is
    rows ``chunk_start[c] .. chunk_start[c] + chunk_len[c]``;
  * matrices are bf16 bit patterns (uint16) stored [out, in]; vectors fp32.
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from dataclasses import dataclass, field, replace
from typing import Dict, List, Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libcrfixtures.so")
_SRC = os.path.join(_HERE, "gen.c")
_lock = threading.Lock()
_lib_handle = None


def build_fixtures(force: bool = False) -> str:
    """Compile gen.c into a shared library (plain gcc, OpenMP). Returns the path."""
    os.makedirs(_BUILD, exist_ok=True)
    if not force and os.path.exists(_SO) and os.path.getmtime(_SO) >= os.path.getmtime(_SRC):
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fopenmp", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _lib():
    global _lib_handle
    with _lock:
        if _lib_handle is None:
            lib = ctypes.CDLL(build_fixtures())
            u64, i64, vp = ctypes.c_uint64, ctypes.c_int64, ctypes.c_void_p
            lib.fx_bits.argtypes = [u64, u64, u64, i64, vp]
            lib.fx_unit_f64.argtypes = [u64, u64, u64, i64, vp]
            lib.fx_normal_rows.argtypes = [u64, u64, i64, i64, i64, ctypes.c_double, vp,
                                           ctypes.c_int, vp]
            lib.fx_uniform_sym.argtypes = [u64, u64, i64, ctypes.c_double, ctypes.c_int, vp]
            lib.fx_f32_to_bf16.argtypes = [vp, i64, vp]
            for f in (lib.fx_bits, lib.fx_unit_f64, lib.fx_normal_rows, lib.fx_uniform_sym,
                      lib.fx_f32_to_bf16):
                f.restype = None
            _lib_handle = lib
        return _lib_handle


def stream_id(name: str) -> int:
    """Stable 64-bit stream id for a tensor name (FNV-1a)."""
    h = 0xCBF29CE484222325
    for b in name.encode():
        h = ((h ^ b) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    return h


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


# ---------------------------------------------------------------- dtype helpers
def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    return bf16_to_f32(bits).astype(np.float64)


def f32_to_bf16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, np.uint16)
    _lib().fx_f32_to_bf16(_ptr(x), x.size, _ptr(out))
    return out


def unit_draws(seed: int, name: str, n: int, offset: int = 0) -> np.ndarray:
    out = np.empty(n, np.float64)
    _lib().fx_unit_f64(seed, stream_id(name), offset, n, _ptr(out))
    return out


def normal_rows(seed: int, name: str, row0: int, n_rows: int, width: int, scale: float = 1.0,
                col_scale: Optional[np.ndarray] = None, dtype: str = "bf16") -> np.ndarray:
    """[n_rows, width] normal draws, row-indexed so any row range regenerates identically."""
    code = 0 if dtype == "f32" else 1
    out = np.empty((n_rows, width), np.float32 if code == 0 else np.uint16)
    cs = None
    if col_scale is not None:
        cs = np.ascontiguousarray(col_scale, dtype=np.float32)
        assert cs.shape == (width,)
    _lib().fx_normal_rows(seed, stream_id(name), row0, n_rows, width, float(scale),
                          None if cs is None else _ptr(cs), code, _ptr(out))
    return out


def xavier_bf16(seed: int, name: str, shape: Sequence[int], fan_in: int, fan_out: int) -> np.ndarray:
    """Xavier-uniform U(+-sqrt(6/(fan_in+fan_out))) drawn in fp32, rounded once to bf16."""
    n = int(np.prod(shape))
    out = np.empty(n, np.uint16)
    a = math.sqrt(6.0 / (fan_in + fan_out))
    _lib().fx_uniform_sym(seed, stream_id(name), n, a, 1, _ptr(out))
    return out.reshape(shape)


def uniform_f32(seed: int, name: str, n: int, a: float, center: float = 0.0) -> np.ndarray:
    out = np.empty(n, np.float32)
    _lib().fx_uniform_sym(seed, stream_id(name), n, a, 0, _ptr(out))
    return (out + np.float32(center)).astype(np.float32)


# ---------------------------------------------------------------- dimensions
@dataclass(frozen=True)
class TargetDims:
    n_layers: int
    n_kv_heads: int
    head_dim: int
    d_model: int
    cache_dtype: str = "bf16"       # "bf16" or "f32"
    rope_theta: float = 1e4         # target LLM RoPE base (global RoPE on repaired K)

    @property
    def n_segments(self) -> int:    # S = 2 L H_kv  (Section 4.1, StaleEncoder)
        return 2 * self.n_layers * self.n_kv_heads

    @property
    def d_kv(self) -> int:          # D_KV = S d_h
        return self.n_segments * self.head_dim


@dataclass(frozen=True)
class RepairerDims:
    d_seg: int
    d_c: int
    d_b: int
    n_blocks: int
    n_heads: int
    mlp_hidden: int
    ln_eps: float = 1e-5
    rope_theta: float = 1e4         # repairer's own RoPE on attention Q/K

    @property
    def head_dim(self) -> int:
        return self.d_b // self.n_heads


@dataclass
class ChunkPlan:
    """Pool layout and the per-request chunk selection (host arrays)."""
    chunk_len: np.ndarray            # int32 [n_pool_chunks]
    chunk_start: np.ndarray          # int64 [n_pool_chunks]
    chunk_idx: np.ndarray            # int32 [sum of chunks over requests]
    cu_chunks: np.ndarray            # int32 [n_req + 1]

    @property
    def n_pool_tokens(self) -> int:
        return int(self.chunk_start[-1] + self.chunk_len[-1]) if len(self.chunk_len) else 0

    def request_lengths(self) -> List[int]:
        out = []
        for r in range(len(self.cu_chunks) - 1):
            sel = self.chunk_idx[self.cu_chunks[r]:self.cu_chunks[r + 1]]
            out.append(int(self.chunk_len[sel].sum()))
        return out

    @property
    def n_tokens(self) -> int:
        return int(sum(self.request_lengths()))


@dataclass
class Recipe:
    """How one workload's inputs are drawn (values, scales, chunk structure)."""
    name: str
    seed: int
    target: TargetDims
    repairer: RepairerDims
    kv_scale: float = 1.0                  # global std of the stale cache
    per_layer_scale: bool = False          # std_l ~ U(0.5, 2) per target layer
    k_outlier_frac: float = 0.0            # fraction of K coordinates scaled x8
    emb_std: float = 0.02
    random_affine: bool = False            # nonzero biases and LN affine (tests only)
    # chunk structure: either explicit request chunk lengths or a pool draw
    pool_lengths: Optional[List[int]] = None
    pool_len_range: Optional[tuple] = None  # (lo, hi) inclusive, drawn per pool chunk
    n_pool_chunks: int = 0
    requests: Optional[List[List[int]]] = None   # explicit pool-chunk indices per request
    n_req_chunks: Optional[int] = None            # single request: draw this many chunks
    batched: Optional[dict] = None                # {"n_req", "lo", "hi", "tok_lo", "tok_hi"}


def _rng(seed: int, name: str) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(key=[seed, stream_id(name) & 0xFFFFFFFFFFFFFFFF]))


def plan_chunks(rc: Recipe) -> ChunkPlan:
    g = _rng(rc.seed, "chunk_plan")
    if rc.pool_lengths is not None:
        lens = np.asarray(rc.pool_lengths, np.int32)
    else:
        lo, hi = rc.pool_len_range
        lens = g.integers(lo, hi + 1, size=rc.n_pool_chunks).astype(np.int32)
    starts = np.zeros(len(lens), np.int64)
    starts[1:] = np.cumsum(lens[:-1].astype(np.int64))
    if rc.requests is not None:
        reqs = [list(r) for r in rc.requests]
    elif rc.batched is not None:
        b = rc.batched
        reqs = []
        for _ in range(b["n_req"]):
            while True:       # redraw until the request length lands in the stated band
                k = int(g.integers(b["lo"], b["hi"] + 1))
                sel = g.choice(len(lens), size=k, replace=False)
                tot = int(lens[sel].sum())
                if b["tok_lo"] <= tot <= b["tok_hi"]:
                    break
            reqs.append([int(x) for x in sel])
    else:
        reqs = [[int(x) for x in g.choice(len(lens), size=rc.n_req_chunks, replace=False)]]
    idx = np.asarray([c for r in reqs for c in r], np.int32)
    cu = np.zeros(len(reqs) + 1, np.int32)
    cu[1:] = np.cumsum([len(r) for r in reqs])
    return ChunkPlan(chunk_len=lens, chunk_start=starts, chunk_idx=idx, cu_chunks=cu)


def sigma_stale_for(rc: Recipe) -> np.ndarray:
    """Per-coordinate std of the synthetic stale cache ([D_KV] fp32).

    The generator draws kv[t, j] = sigma[j] * N(0,1); sigma is therefore the
    exact RMS the paper's sigma_stale estimates (Section 4.2, "Normalization").
    """
    t = rc.target
    L, H, dh = t.n_layers, t.n_kv_heads, t.head_dim
    sig = np.full((L, 2, H, dh), rc.kv_scale, np.float64)
    if rc.per_layer_scale:
        g = _rng(rc.seed, "layer_scale")
        sig *= g.uniform(0.5, 2.0, size=L)[:, None, None, None]
    if rc.k_outlier_frac > 0:
        g = _rng(rc.seed, "k_outliers")
        n_k = L * H * dh
        n_out = int(round(rc.k_outlier_frac * n_k))
        pick = g.choice(n_k, size=n_out, replace=False)
        kview = sig[:, 0].reshape(-1)          # copy of the K coordinates
        kview[pick] *= 8.0
        sig[:, 0] = kview.reshape(L, H, dh)
    return sig.reshape(-1).astype(np.float32)


def inv_freq_for(theta: float, dim: int) -> np.ndarray:
    """RoPE inverse frequencies theta^(-2i/dim), i < dim/2, as fp32 (a target-model input)."""
    i = np.arange(dim // 2, dtype=np.float64)
    return (theta ** (-2.0 * i / dim)).astype(np.float32)


# sigma_Delta = RESIDUAL_SCALE * sigma_stale.  The residual the method adds is
# sigma_Delta * z with z = W_out y_f + b_out; with LN_f's unit-variance y_f and
# the Xavier head (d_b -> D_KV) std(z) = sqrt(2 d_b / (d_b + D_KV)), about 0.17
# at d_b = 1024, D_KV = 65536.  A scale of 1 makes the residual about 17 % of
# the stale cache (25 % at d_b = 512), the size the paper measures between
# stale and joint caches (Sec. 5.3: relative RMSE 0.18 inside chunks, 0.31 at
# chunk boundaries).
RESIDUAL_SCALE = 1.0


def make_weights(rc: Recipe) -> Dict[str, np.ndarray]:
    """Random-init repairer weights: Xavier-uniform matrices (bf16), biases 0, LN identity.

    Shapes follow Section 4.1: per-segment d_h->d_seg projections, the map
    S*d_seg -> d_c, P_tok d_model -> d_c, F 2d_c -> d_b, one P_b d_c -> d_b per
    block, B pre-LN blocks, final LN, KV residual head d_b -> D_KV.
    """
    t, p, s = rc.target, rc.repairer, rc.seed
    S, dh, D = t.n_segments, t.head_dim, t.d_kv
    db, dc, ds, B, hid = p.d_b, p.d_c, p.d_seg, p.n_blocks, p.mlp_hidden
    w: Dict[str, np.ndarray] = {}

    def vec(name, n, kind):
        if not rc.random_affine:
            return np.ones(n, np.float32) if kind == "gamma" else np.zeros(n, np.float32)
        if kind == "gamma":
            return uniform_f32(s, name, n, 0.25, center=1.0)
        return uniform_f32(s, name, n, 0.1)

    w["w_seg"] = xavier_bf16(s, "w_seg", (S, ds, dh), dh, ds)
    w["b_seg"] = vec("b_seg", S * ds, "bias").reshape(S, ds)
    w["w_map"] = xavier_bf16(s, "w_map", (dc, S * ds), S * ds, dc)
    w["b_map"] = vec("b_map", dc, "bias")
    w["w_tok"] = xavier_bf16(s, "w_tok", (dc, t.d_model), t.d_model, dc)
    w["b_tok"] = vec("b_tok", dc, "bias")
    w["w_fuse"] = xavier_bf16(s, "w_fuse", (db, 2 * dc), 2 * dc, db)
    w["b_fuse"] = vec("b_fuse", db, "bias")
    w["w_rein"] = np.stack([xavier_bf16(s, f"w_rein{b}", (db, dc), dc, db) for b in range(B)]) \
        if B else np.zeros((0, db, dc), np.uint16)
    w["b_rein"] = np.stack([vec(f"b_rein{b}", db, "bias") for b in range(B)]) \
        if B else np.zeros((0, db), np.float32)
    for b in range(B):
        w[f"blk{b}.ln1_g"] = vec(f"blk{b}.ln1_g", db, "gamma")
        w[f"blk{b}.ln1_b"] = vec(f"blk{b}.ln1_b", db, "beta")
        w[f"blk{b}.w_qkv"] = xavier_bf16(s, f"blk{b}.w_qkv", (3 * db, db), db, 3 * db)
        w[f"blk{b}.b_qkv"] = vec(f"blk{b}.b_qkv", 3 * db, "bias")
        w[f"blk{b}.w_o"] = xavier_bf16(s, f"blk{b}.w_o", (db, db), db, db)
        w[f"blk{b}.b_o"] = vec(f"blk{b}.b_o", db, "bias")
        w[f"blk{b}.ln2_g"] = vec(f"blk{b}.ln2_g", db, "gamma")
        w[f"blk{b}.ln2_b"] = vec(f"blk{b}.ln2_b", db, "beta")
        w[f"blk{b}.w_fc1"] = xavier_bf16(s, f"blk{b}.w_fc1", (hid, db), db, hid)
        w[f"blk{b}.b_fc1"] = vec(f"blk{b}.b_fc1", hid, "bias")
        w[f"blk{b}.w_fc2"] = xavier_bf16(s, f"blk{b}.w_fc2", (db, hid), hid, db)
        w[f"blk{b}.b_fc2"] = vec(f"blk{b}.b_fc2", db, "bias")
    w["lnf_g"] = vec("lnf_g", db, "gamma")
    w["lnf_b"] = vec("lnf_b", db, "beta")
    w["w_out"] = xavier_bf16(s, "w_out", (D, db), db, D)
    w["b_out"] = vec("b_out", D, "bias")
    sig = sigma_stale_for(rc)
    w["sigma_stale"] = sig
    # sigma_Delta is the per-coordinate RMS of the joint - stale residual (Sec. 4.2);
    # synthetic: the stale cache's own scale (see RESIDUAL_SCALE)
    w["sigma_delta"] = (RESIDUAL_SCALE * sig).astype(np.float32)
    return w


@dataclass
class Case:
    recipe: Recipe
    plan: ChunkPlan
    weights: Dict[str, np.ndarray]
    inv_freq_target: np.ndarray         # [head_dim/2] fp32, target R_M frequencies

    @property
    def target(self) -> TargetDims:
        return self.recipe.target

    @property
    def repairer(self) -> RepairerDims:
        return self.recipe.repairer

    def pool_rows(self, row0: int, n_rows: int):
        """Stale cache and embeddings for pool rows [row0, row0 + n_rows)."""
        rc, t = self.recipe, self.recipe.target
        kv = normal_rows(rc.seed, "kv_pool", row0, n_rows, t.d_kv, 1.0,
                         self.weights["sigma_stale"], t.cache_dtype)
        emb = normal_rows(rc.seed, "emb_pool", row0, n_rows, t.d_model, rc.emb_std,
                          None, t.cache_dtype)
        return kv, emb

    def pool(self):
        return self.pool_rows(0, self.plan.n_pool_tokens)

    def request_pool_rows(self, r: int):
        """Pool rows of request r's chunks in document order (for the oracle)."""
        p = self.plan
        sel = p.chunk_idx[p.cu_chunks[r]:p.cu_chunks[r + 1]]
        kvs, embs = [], []
        for c in sel:
            kv, emb = self.pool_rows(int(p.chunk_start[c]), int(p.chunk_len[c]))
            kvs.append(kv)
            embs.append(emb)
        return sel, kvs, embs


# ---------------------------------------------------------------- the workloads
TINY_T = TargetDims(4, 2, 64, 256, "f32", 1e4)
QWEN3B_T = TargetDims(36, 2, 128, 2048, "bf16", 1e6)
LLAMA8B_T = TargetDims(32, 8, 128, 4096, "bf16", 5e5)
QWEN7B_T = TargetDims(28, 4, 128, 3584, "bf16", 1e6)


def _recipes() -> Dict[str, Recipe]:
    r = {}
    r["tiny"] = Recipe("tiny", 0, TINY_T, RepairerDims(8, 64, 128, 2, 4, 512),
                       kv_scale=0.5, pool_lengths=[64] * 4, n_req_chunks=2)
    r["qwen3b"] = Recipe("qwen3b", 1, QWEN3B_T, RepairerDims(8, 256, 512, 4, 8, 2048),
                         per_layer_scale=True, pool_lengths=[512] * 8, n_req_chunks=5)
    r["llama8b"] = Recipe("llama8b", 2, LLAMA8B_T, RepairerDims(16, 512, 1024, 6, 16, 4096),
                          per_layer_scale=True, k_outlier_frac=0.01,
                          pool_lengths=[512] * 12, n_req_chunks=10)
    r["qwen7b"] = Recipe("qwen7b", 3, QWEN7B_T, RepairerDims(16, 512, 1024, 8, 16, 4096),
                         per_layer_scale=True, pool_len_range=(128, 512), n_pool_chunks=24,
                         n_req_chunks=20)
    r["batched"] = Recipe("batched", 4, LLAMA8B_T, RepairerDims(16, 512, 1024, 6, 16, 4096),
                          pool_len_range=(64, 1024), n_pool_chunks=256,
                          batched=dict(n_req=16, lo=4, hi=16, tok_lo=6144, tok_hi=10240))
    # Test-only shapes: several 128-row tiles with ragged tails, a 1-token chunk,
    # nonzero biases and LN affine so that every epilogue term is exercised.
    small_t = TargetDims(4, 2, 128, 512, "bf16", 1e6)
    small_r = RepairerDims(8, 128, 256, 2, 4, 1024)
    r["small"] = Recipe("small", 11, small_t, small_r, per_layer_scale=True,
                        k_outlier_frac=0.01, random_affine=True,
                        pool_lengths=[130, 77, 200, 1, 95, 64], requests=[[2, 0, 3, 1, 4]])
    r["small_multi"] = Recipe("small_multi", 12, small_t, small_r, per_layer_scale=True,
                              random_affine=True,
                              pool_lengths=[130, 77, 200, 1, 95, 64, 300, 33],
                              requests=[[1, 2], [6], [7, 3, 0, 5]])
    r["tiny_affine"] = replace(r["tiny"], name="tiny_affine", seed=5, random_affine=True)
    return r


RECIPES: Dict[str, Recipe] = _recipes()
WORKLOAD_CONFIGS = ["tiny", "qwen3b", "llama8b", "qwen7b", "batched"]


def make_case(name_or_recipe, **overrides) -> Case:
    rc = RECIPES[name_or_recipe] if isinstance(name_or_recipe, str) else name_or_recipe
    if overrides:
        rc = replace(rc, **overrides)
    plan = plan_chunks(rc)
    w = make_weights(rc)
    return Case(rc, plan, w, inv_freq_for(rc.target.rope_theta, rc.target.head_dim))
