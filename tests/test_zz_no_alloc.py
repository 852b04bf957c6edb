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
from gpu_util import grad_rel_err

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
        torch.cuda.synchronize()
        assert grad_rel_err(got.cpu().numpy(), ref) <= 1e-3


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
