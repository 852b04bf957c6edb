"""The dense tensor-core rate kernels (the contractions' roofline
denominators) run, drain and report their operation counts."""
import pytest
import torch

from paper_2010_14298_gb300 import fqt

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="no GPU")]


@pytest.mark.parametrize("kind,per_iter", [(0, 2 * 128 * 256 * 16 * 4),
                                           (1, 2 * 128 * 256 * 32 * 4)])
def test_tcgen05_rate_kernels(kind, per_iter):
    ws = fqt.Workspace(1, 16, 16)
    ops = fqt.debug_mma_peak(kind, 64, ws)
    assert fqt.sync_status(ws) == 0
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    assert ops == per_iter * 64 * sms


def test_imma_rate_kernel():
    ws = fqt.Workspace(1, 16, 16)
    ops = fqt.debug_mma_peak(2, 16, ws)
    assert fqt.sync_status(ws) == 0
    assert ops > 0


def test_rate_kernel_arguments():
    ws = fqt.Workspace(1, 16, 16)
    for kind, iters in ((3, 1), (0, 0), (-1, 5)):
        with pytest.raises(fqt.FqtError) as e:
            fqt.debug_mma_peak(kind, iters, ws)
        assert e.value.status == 1
