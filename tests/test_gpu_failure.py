"""Failure detection without faulting the GPU: a bounded device wait that nothing
completes reports CS_ERR_TIMEOUT through cs_sync_status, and the context stays usable."""
import numpy as np
import pytest
import torch

import oracle as O
from _helpers import cuda, f64

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_survives(cslib):
    cslib.cs_sync_status()
    cslib.cs_debug_wait_timeout(20000)          # 20 ms
    with pytest.raises(cslib.CsError) as e:
        cslib.cs_sync_status()
    assert e.value.status == cslib.CS_ERR_TIMEOUT
    cslib.cs_sync_status()                      # the status word was cleared
    # the context still runs kernels correctly
    s = torch.tensor([3.0, 1.0, 2.0, 5.0], device="cuda")
    idx = cslib.cs_select_topk(s, 2, 10)
    cslib.cs_sync_status()
    assert idx.cpu().tolist() == [10, 13]
    k = torch.randn((1, 8, 2, 128), device="cuda").to(torch.bfloat16)
    loc = np.zeros((8, 3), np.int32)
    glo = np.tile(np.array([[5, 6, 7]], np.int32), (8, 1))
    before = f64(k)
    cslib.cs_rebase_keys(k, cuda(loc), cuda(glo))
    cslib.cs_sync_status()
    exp, _ = O.rebase(before, loc, glo, "bf16")
    assert np.array_equal(f64(k), exp)


def test_status_record_is_device_wide_and_taken_once(cslib):
    """An error recorded by a kernel on one stream is reported by the next take on any
    stream of the device (the record is device-wide), exactly once."""
    cslib.cs_sync_status()
    a, b = torch.cuda.Stream(), torch.cuda.Stream()
    cslib.cs_debug_wait_timeout(20000, stream=a)   # records CS_ERR_TIMEOUT on stream a
    a.synchronize()
    with pytest.raises(cslib.CsError) as e:
        cslib.cs_sync_status(stream=b)
    assert e.value.status == cslib.CS_ERR_TIMEOUT
    cslib.cs_sync_status(stream=a)                  # taken already: nothing left
    cslib.cs_sync_status(stream=b)
