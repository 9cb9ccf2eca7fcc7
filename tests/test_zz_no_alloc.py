"""cr_segment_project_noalloc: the segment projection for callers that cannot
allocate device memory (no workspace argument; its scratch is a fixed array
inside the library).  Its output must match cr_segment_project, which takes a
caller workspace, on two calls in a row with different inputs.  This file runs
last so that, if it fails, a run stopping at the first failure has already run
every other test."""
import numpy as np
import pytest
import torch

import fixtures as F
from paper_2609_35139_gb300 import build, cr, dims_from
from parity_util import assert_close, to_dev, to_host

pytestmark = pytest.mark.gpu


def test_noalloc_segment_projection_matches_workspace_version():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    cr.lib()
    for call, (name, row0) in enumerate([("llama8b", 0), ("qwen3b", 300)]):
        c = F.make_case(name)
        t, r = c.target, c.repairer
        td, _ = dims_from(t, r)
        kv, _ = c.pool_rows(row0, 600)
        w = c.weights
        args = (to_dev(kv), to_dev(w["w_seg"]), to_dev(w["b_seg"]), to_dev(w["sigma_stale"]))
        width = t.n_segments * r.d_seg
        y_ws = torch.empty(600, width, dtype=torch.bfloat16, device="cuda")
        ws = torch.empty(t.n_segments * r.d_seg * t.head_dim * 4, dtype=torch.uint8, device="cuda")
        cr.cr_segment_project(td, r.d_seg, *args, y_ws, ws)
        y_na = torch.full((600, width), float("nan"), dtype=torch.bfloat16, device="cuda")
        cr.cr_segment_project_noalloc(td, r.d_seg, *args, y_na)
        torch.cuda.synchronize()
        a, b = to_host(y_na), to_host(y_ws)
        assert_close(a, b, 1e-6, 1e-5, f"no-alloc vs workspace, call {call + 1} ({name})")
    st, word = cr.cr_get_device_status()
    assert st == cr.CR_OK, word


def test_noalloc_rejects_oversized_shapes():
    """Shapes whose weights exceed the fixed scratch (2 Mi weights, two bf16 terms each:
    8 MiB) are refused on the host, including L * H_kv so large that S * d_seg * d_h
    would not fit in 64 bits; target dimensions are checked as cr_segment_project
    checks them."""
    build.build()
    FAKE = 0x10000
    L = cr.lib()
    import ctypes

    def call(t, d_seg=16):
        return L.cr_segment_project_noalloc(ctypes.byref(t), d_seg, FAKE, 10, FAKE, FAKE, FAKE, FAKE,
                                            None)

    assert call(cr.target_dims(80, 16, 128, 8192, "bf16")) == cr.CR_ERR_UNSUPPORTED   # 5 Mi weights
    assert call(cr.target_dims(2 ** 30, 2 ** 30, 128, 8192, "bf16")) == cr.CR_ERR_UNSUPPORTED
    assert call(cr.target_dims(4, 2, 128, 0, "bf16")) == cr.CR_ERR_INVALID_ARG       # d_model
    assert call(cr.target_dims(4, 2, 128, 4096, 7)) == cr.CR_ERR_INVALID_ARG         # cache dtype
    assert call(cr.target_dims(4, 2, 96, 4096, "bf16")) == cr.CR_ERR_UNSUPPORTED     # head dim
    assert call(cr.target_dims(4, 2, 128, 4096, "bf16"), d_seg=12) == cr.CR_ERR_UNSUPPORTED
