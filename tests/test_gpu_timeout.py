"""The device-side timeout path, without faulting or hanging the GPU.

A kernel waits on an mbarrier that nothing arrives at, with the same bounded
wait the contraction kernels use and a short limit.  It must return, record
FQT_ETIMEOUT in the workspace's status word (read once by fqt_sync_status,
then cleared), and leave the context usable for the next call.
"""
import time

import numpy as np
import pytest
import torch

import oracle as orc
from paper_2010_14298_gb300 import fqt
from paper_2010_14298_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="no GPU")]


@pytest.mark.parametrize("limit_ms", [5, 50])
def test_wait_that_runs_out_reports_timeout(limit_ms):
    ws = fqt.Workspace(64, 64, 16)
    assert fqt.sync_status(ws) == 0
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    fqt.debug_wait_timeout(limit_ms * 1_000_000, ws)
    st = fqt.sync_status(ws)
    dt = time.perf_counter() - t0
    assert st == 5, fqt.status_string(st)  # FQT_ETIMEOUT
    assert dt >= limit_ms * 1e-3 * 0.9
    assert dt < limit_ms * 1e-3 + 2.0
    assert fqt.sync_status(ws) == 0  # read once, then cleared
    # the context is still usable: a quantizer call after the timeout is exact
    L = wl.config(0, rows=32)[0]
    q2, _ = fqt.quantize_grad(torch.from_numpy(L.dH).cuda(), fqt.PSQ, 8, 0, 7,
                              with_b1=False, ws=ws)
    assert fqt.sync_status(ws) == 0
    ref = orc.quantize_grad(L.dH, orc.PSQ, 8, 0, 7, orc.STREAM_B2)
    assert np.array_equal(q2.codes.cpu().numpy(), ref["codes"])
