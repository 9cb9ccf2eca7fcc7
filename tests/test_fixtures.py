"""The shared input generator: deterministic, row-addressable, right statistics."""
import numpy as np

import fixtures as F


def test_generator_is_deterministic_and_row_addressable():
    c = F.make_case("small")
    kv, emb = c.pool()
    kv2, emb2 = c.pool_rows(100, 57)
    assert np.array_equal(kv[100:157], kv2) and np.array_equal(emb[100:157], emb2)
    c2 = F.make_case("small")
    assert np.array_equal(c2.pool()[0], kv)
    for k in c.weights:
        assert np.array_equal(c.weights[k], c2.weights[k])


def test_statistics_and_no_negative_zero():
    c = F.make_case("qwen3b")
    kv, emb = c.pool_rows(0, 256)
    x = F.bf16_to_f32(kv).astype(np.float64) / c.weights["sigma_stale"]
    assert abs(x.std() - 1.0) < 0.01 and abs(x.mean()) < 0.01
    assert abs(F.bf16_to_f32(emb).std() - 0.02) < 0.001
    assert not np.any(kv == 0x8000) and not np.any(c.weights["w_out"] == 0x8000)
    w = F.bf16_to_f32(c.weights["w_out"]).astype(np.float64)
    a = np.sqrt(6.0 / (512 + c.target.d_kv))
    assert np.abs(w).max() <= a * 1.004 and abs(w.std() - a / np.sqrt(3)) < 0.01 * a


def test_recipes_match_the_stated_workloads():
    c = F.make_case("llama8b")
    assert c.plan.request_lengths() == [5120] and c.target.d_kv == 65536
    s = c.weights["sigma_stale"].reshape(32, 2, 8, 128)
    k_out = (s[:, 0] / s[:, 1]).reshape(-1)
    assert np.sum(np.isclose(k_out, 8.0)) == round(0.01 * 32 * 8 * 128)
    b = F.make_case("batched")
    lens = b.plan.request_lengths()
    assert len(lens) == 16 and all(6144 <= n <= 10240 for n in lens)
    cpr = np.diff(b.plan.cu_chunks)
    assert cpr.min() >= 4 and cpr.max() <= 16
    for r in range(16):
        sel = b.plan.chunk_idx[b.plan.cu_chunks[r]:b.plan.cu_chunks[r + 1]]
        assert len(set(sel.tolist())) == len(sel)
    s7 = F.make_case("qwen7b")
    sel = s7.plan.chunk_idx
    assert len(sel) == 20 and s7.plan.chunk_len.min() >= 128 and s7.plan.chunk_len.max() <= 512
    t = F.make_case("tiny")
    assert t.plan.request_lengths() == [128] and t.target.cache_dtype == "f32"
