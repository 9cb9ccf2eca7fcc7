"""Failure reporting on the GPU without a fault: a bounded wait that nothing
satisfies gives up, the host reads the timeout from the device status word, and
the context keeps working."""
import numpy as np
import pytest
import torch

from paper_2609_35139_gb300 import build, cr
from parity_util import to_dev, to_host

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_the_context_survives():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    cr.lib()
    cr.cr_clear_device_status()
    cr.cr_wait_selftest()
    st, word = cr.cr_get_device_status()          # synchronises: about 2 s of waiting
    assert st == cr.CR_ERR_TIMEOUT, (st, word)
    assert list(word[:2]) == [1, 900], word
    cr.cr_clear_device_status()
    assert cr.cr_get_device_status()[0] == cr.CR_OK
    # the next call runs and is right
    cend = np.repeat(np.array([3, 3, 3, 7, 7, 7, 7, 8], np.int32), 1)
    out = torch.full((8,), -1, dtype=torch.int32, device="cuda")
    cr.cr_chunk_starts(to_dev(cend), np.array([0, 8], np.int32), 8, out)
    torch.cuda.synchronize()
    assert to_host(out).tolist() == [0, 0, 0, 3, 3, 3, 3, 7]
    assert cr.cr_get_device_status()[0] == cr.CR_OK
