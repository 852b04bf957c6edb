"""fqt_grad_w_fixed_scratch: grad_W for callers that cannot allocate.

Some callers of this library cannot allocate device memory when they run
the backward (a loop whose memory budget is frozen after warm-up, or a plain
C host without an allocator of its own that must not call cudaMalloc).  The
fixed-scratch entry point takes no workspace and keeps its split-K partials
in an array inside the library.  These tests call it through the C ABI and
check it against fqt_linear_backward, twice in a row (the array keeps the
previous call's contents), at sizes where the split plan fits the array and
where it has to be narrowed.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

from paper_2010_14298_gb300 import fqt
from paper_2010_14298_gb300 import workloads as wl

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="no GPU")]


def _operands(cfg, batch, seed=5):
    L = wl.config(cfg, batch=batch)[0]
    qx = fqt.quantize_act(torch.from_numpy(L.X).cuda(), 8)
    _, q1 = fqt.quantize_grad(torch.from_numpy(L.dH).cuda(), fqt.BHQ, 5, 16, seed)
    return L, q1, qx


@pytest.mark.parametrize("cfg,batch", [(1, 2), (2, 16), (2, 1)])
def test_fixed_scratch_matches_workspace_path(cfg, batch):
    L, q1, qx = _operands(cfg, batch)
    ws = fqt.Workspace(L.N, L.C, L.D)
    qw = fqt.quantize_weight(torch.from_numpy(L.W).cuda(), 8)
    q2, _ = fqt.quantize_grad(torch.from_numpy(L.dH).cuda(), fqt.PSQ, 5, 0, 1,
                              with_b1=False)
    _, ref = fqt.linear_backward(q2, q1, qx, qw, grad_x=False, grad_w=True, ws=ws)
    ref = ref.cpu().numpy()
    for _ in range(2):  # the second call sees the first call's leftovers
        got = fqt.grad_w_fixed_scratch(q1, qx)
        assert fqt.fixed_scratch_sync_status() == 0
        # exact int32 partials reduced in int64 then one fixed dequantization:
        # whatever the split plan, the result is the same to the bit
        assert np.array_equal(got.cpu().numpy(), ref)


def test_fixed_scratch_rejects_problems_beyond_its_limit():
    # 2048 x 1152 int32 partials: 9.4 MB per split, more than the 8 MiB array
    C, D, N = 2048, 1152, 64
    g = wl.rng(3)
    qx = fqt.quantize_act(torch.from_numpy(
        g.uniform(-1, 1, (N, D)).astype(np.float32)).cuda(), 8)
    _, q1 = fqt.quantize_grad(torch.from_numpy(
        g.standard_normal((N, C)).astype(np.float32)).cuda(), fqt.PTQ, 8, 0, 0)
    with pytest.raises(fqt.FqtError) as e:
        fqt.grad_w_fixed_scratch(q1, qx)
    assert e.value.status == 6  # FQT_EWORKSPACE


def test_fixed_scratch_refuses_an_implicit_im2col_operand():
    """An operand from quantize_act_conv stores NHWC codes, not the N x D
    matrix the fixed-scratch kernel reads; the call refuses it before any
    launch."""
    g = wl.rng(11)
    X = torch.from_numpy(g.uniform(-1, 1, (2, 32, 32, 64)).astype(np.float32)).cuda()
    qx = fqt.quantize_act_conv(X, 3, 3, 1, 8)
    _, q1 = fqt.quantize_grad(torch.from_numpy(
        g.standard_normal((qx.shape[0], 64)).astype(np.float32)).cuda(), fqt.PTQ, 8, 0, 0)
    out = torch.full((64, qx.shape[1]), 7.0, device="cuda")
    with pytest.raises(fqt.FqtError) as e:
        fqt.grad_w_fixed_scratch(q1, qx, out=out)
    assert e.value.status == 2  # FQT_EUNSUPPORTED
    assert bool((out == 7.0).all())  # nothing was written


def test_fixed_scratch_status_reports_a_wait_that_ran_out():
    """A bounded wait made to run out records FQT_ETIMEOUT in the fixed
    array's status word; the reader returns it once, then FQT_OK, and the
    entry point still computes afterwards."""
    assert fqt.fixed_scratch_sync_status() == 0
    fqt.debug_wait_timeout(20_000_000)  # 20 ms, nothing arrives
    assert fqt.fixed_scratch_sync_status() == 5  # FQT_ETIMEOUT
    assert fqt.fixed_scratch_sync_status() == 0
    L, q1, qx = _operands(1, 2)
    got = fqt.grad_w_fixed_scratch(q1, qx)
    assert fqt.fixed_scratch_sync_status() == 0
    assert torch.isfinite(got).all()
