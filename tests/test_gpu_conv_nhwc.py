"""grad_X of a stride-1 3x3 conv in NHWC with col2im fused into the
contraction (fqt_conv_grad_x_nhwc), against the oracle's col2im of its
dequantize-then-multiply (Sec. 2.1, Eq. 6) fed the GPU's codes.  Q_b2 is
per tensor (PTQ) or per image (PSQ with one sample per image, Sec. 4.1)."""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2010_14298_gb300 import fqt
from paper_2010_14298_gb300 import workloads as wl
from gpu_util import grad_rel_err, to_dev

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="no GPU")]

CASES = [  # n, h, w, cin, cout, kind, bits
    (2, 32, 32, 64, 64, orc.PSQ, 5), (2, 32, 32, 64, 64, orc.PTQ, 8),
    (1, 56, 56, 64, 64, orc.PSQ, 5), (2, 28, 28, 128, 128, orc.PSQ, 5),
    (2, 14, 14, 256, 256, orc.PSQ, 5), (3, 7, 7, 512, 512, orc.PSQ, 5),
    (2, 9, 10, 96, 64, orc.PTQ, 4), (1, 2, 2, 32, 64, orc.PSQ, 8)]


def _operands(n, h, w, cin, cout, kind, bits, seed=7):
    g = wl.rng(n * 1000 + h * 10 + cin + cout)
    dH = wl.random_grad(g, n * h * w, cout, sigma=1.0)
    dH *= np.repeat(np.exp(1.5 * g.standard_normal(n)), h * w)[:, None].astype(np.float32)
    W = (np.sqrt(2.0 / (9 * cin)) * g.standard_normal((cout, 9 * cin))).astype(np.float32)
    qw = fqt.quantize_weight(to_dev(W), 8)
    if kind == orc.PSQ:
        q2, _ = fqt.quantize_grad_samples(to_dev(dH), h * w, orc.PSQ, bits, seed=seed,
                                          with_b1=False)
    else:
        q2, _ = fqt.quantize_grad(to_dev(dH), orc.PTQ, bits, 0, seed, with_b1=False)
    return dH, W, q2, qw


def _oracle(q2, qw, n, h, w, cin, kind):
    h2 = q2.to_numpy()
    if kind == orc.PSQ:
        R = h * w
        h2 = dict(h2, inv_s=h2["inv_s"][::R], zero=h2["zero"][::R], rows_per_sample=R)
    return orc.grad_x_nhwc(h2, qw.to_numpy(), n, h, w, cin, 3, 1)


@pytest.mark.parametrize("n,h,w,cin,cout,kind,bits", CASES)
def test_conv_grad_x_nhwc_matches_oracle(n, h, w, cin, cout, kind, bits):
    dH, W, q2, qw = _operands(n, h, w, cin, cout, kind, bits)
    ws = fqt.Workspace(1, 16, 16)
    ws.nbytes = int(fqt.load().fqt_conv_grad_x_workspace_size(cin))
    ws.buf = torch.zeros(ws.nbytes, dtype=torch.uint8, device="cuda")
    out = fqt.conv_grad_x_nhwc(q2, qw, n, h, w, cin, ws=ws)
    assert fqt.sync_status(ws) == 0
    ref = _oracle(q2, qw, n, h, w, cin, kind)
    got = out.cpu().numpy()
    assert np.isfinite(got).all()
    assert grad_rel_err(got.reshape(-1, cin), ref.reshape(-1, cin)) <= 1e-3


def test_fused_col2im_equals_col2im_of_the_im2col_grad_x():
    """The NHWC contraction against col2im of the im2col-space grad_X of
    fqt_linear_backward on the same codes (two GPU paths, one layer)."""
    n, h, w, cin, cout = 2, 32, 32, 64, 64
    dH, W, q2, qw = _operands(n, h, w, cin, cout, orc.PSQ, 5)
    out = fqt.conv_grad_x_nhwc(q2, qw, n, h, w, cin)
    gx, _ = fqt.linear_backward(q2, None, None, qw, grad_x=True, grad_w=False)
    torch.cuda.synchronize()
    ref = orc.col2im_nhwc(gx.cpu().numpy().astype(np.float64), n, h, w, cin, 3, 3, 1, 1)
    assert grad_rel_err(out.cpu().numpy().reshape(-1, cin), ref.reshape(-1, cin)) <= 1e-4


def test_conv_grad_x_nhwc_refusals():
    n, h, w, cin, cout = 1, 8, 8, 32, 64
    dH, W, q2, qw = _operands(n, h, w, cin, cout, orc.PSQ, 5)
    with pytest.raises(fqt.FqtError) as e:
        fqt.conv_grad_x_nhwc(q2, qw, n, h, w, cin, k=5, pad=2)
    assert e.value.status == 2
    # per-row PSQ: the scale is not constant over an image
    q_rows, _ = fqt.quantize_grad(to_dev(dH), orc.PSQ, 5, 0, 1, with_b1=False)
    with pytest.raises(fqt.FqtError) as e:
        fqt.conv_grad_x_nhwc(q_rows, qw, n, h, w, cin)
    assert e.value.status == 2
