"""Offline preparation kernels against the oracle: chunk canonicalisation
(Sec. 4.1) and the sigma statistics (Sec. 4.2)."""
import numpy as np
import pytest
import torch

import fixtures as F
import oracle as O
from paper_2609_35139_gb300 import cr
from parity_util import as_f64, half_ulp, to_dev, to_host

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2609_35139_gb300 import build
    build.build()
    cr.lib()
    cr.cr_clear_device_status()
    yield
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, f"device status {word}"


def _cache(n, L, H, dh, dtype, seed):
    g = np.random.default_rng(seed)
    x = (g.standard_normal((n, 2 * L * H * dh)) * 2.0).astype(np.float32)
    return F.f32_to_bf16(x) if dtype == "bf16" else x


def _local_positions(lens, offset=0):
    return np.concatenate([np.arange(n) + offset for n in lens]).astype(np.int32)


@pytest.mark.parametrize("L,H,dh,dtype,theta,offset", [
    (4, 2, 128, "bf16", 1e6, 0),        # chunk-local positions
    (32, 8, 128, "bf16", 5e5, 3000),    # 8B shape, large positions
    (4, 2, 64, "f32", 1e4, 0),
])
def test_canonicalize_matches_oracle(L, H, dh, dtype, theta, offset):
    lens = [130, 77, 1, 126]
    n = sum(lens)
    kv = _cache(n, L, H, dh, dtype, seed=L + dh)
    pos = _local_positions(lens, offset)
    inv = (theta ** (-np.arange(0, dh, 2) / dh)).astype(np.float32)
    t = cr.target_dims(L, H, dh, 256, dtype)
    dev = to_dev(kv)
    cr.cr_canonicalize_chunks(t, dev, n, to_dev(pos), inv)
    torch.cuda.synchronize()
    got = to_host(dev)
    ref = O.canonicalize_chunk(kv, pos, inv, n_layers=L, n_kv_heads=H, head_dim=dh, cache_dtype=dtype)
    v = lambda a: a.reshape(n, L, 2, H, dh)[:, :, 1]
    assert np.array_equal(v(got), v(kv))                       # V untouched
    # bound: one rounding of the exact value (half an ulp of the cache dtype)
    # plus the fp32 evaluation of the rotation, relative to the pair's size
    # |a| + |b| (which is what a cancellation near zero leaves as error)
    exact = O.canonical_exact(kv, pos, inv, n_layers=L, n_kv_heads=H, head_dim=dh, cache_dtype=dtype)
    x = (as_f64(kv) if dtype == "bf16" else kv.astype(np.float64)).reshape(n, L, 2, H, dh)[:, :, 0]
    mag = np.abs(x[..., : dh // 2]) + np.abs(x[..., dh // 2:])
    mag = np.concatenate([mag, mag], axis=-1)
    k = lambda a: a.reshape(n, L, 2, H, dh)[:, :, 0]
    g = k(as_f64(got) if dtype == "bf16" else got.astype(np.float64))
    e = k(exact)
    err = np.abs(g - e)
    bound = half_ulp(e, dtype) + 2e-6 * mag
    assert np.all(err <= bound), float(np.max(err - bound))
    if dtype == "bf16":
        # and away from cancellation the stored value is the oracle's own rounding
        assert np.mean(got == ref) > 0.99


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_sigma_statistics_match_oracle_and_are_deterministic(dtype):
    L, H, dh = (4, 2, 128) if dtype == "bf16" else (4, 2, 64)
    t = cr.target_dims(L, H, dh, 256, dtype)
    D = 2 * L * H * dh
    batches = [_cache(n, L, H, dh, dtype, seed=i) for i, n in enumerate([100, 64, 257])]
    joints = [_cache(b.shape[0], L, H, dh, dtype, seed=10 + i) for i, b in enumerate(batches)]
    count = sum(b.shape[0] for b in batches)

    def run(with_b):
        sumsq = torch.zeros(D, dtype=torch.float64, device="cuda")
        for a, j in zip(batches, joints):
            n = a.shape[0]
            ws = torch.empty(cr.cr_sigma_workspace_bytes(t, n), dtype=torch.uint8, device="cuda")
            cr.cr_sigma_accumulate(t, to_dev(j) if with_b else to_dev(a), to_dev(a) if with_b else None,
                                   n, sumsq, ws)
        sig = torch.empty(D, dtype=torch.float32, device="cuda")
        cr.cr_sigma_finalize(t, sumsq, count, sig)
        torch.cuda.synchronize()
        return to_host(sig)

    s_stale = run(False)
    np.testing.assert_allclose(s_stale, O.sigma_rms(batches, dtype), rtol=1e-5)
    s_delta = run(True)
    np.testing.assert_allclose(s_delta, O.sigma_rms(joints, dtype, minus=batches), rtol=1e-5)
    assert np.array_equal(run(True).view(np.uint32), s_delta.view(np.uint32))
