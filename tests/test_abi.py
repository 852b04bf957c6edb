"""The C-ABI library builds, loads and exports every entry point that
include/fqt.h declares (no GPU needed: nothing is computed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "fqt.h")


def declared_symbols():
    text = open(HEADER).read()
    return re.findall(r"FQT_API\s+[\w\s\*]*?\b(fqt_\w+)\s*\(", text)


def test_header_declares_the_boundary():
    names = set(declared_symbols())
    for required in ("fqt_quantize_act", "fqt_quantize_weight",
                     "fqt_quantize_grad", "fqt_linear_backward", "fqt_linear_forward",
                     "fqt_quantize_act_conv",
                     "fqt_workspace_size", "fqt_sync_status",
                     "fqt_status_string", "fqt_debug_int_gemm"):
        assert required in names


def test_library_exports_every_declared_symbol():
    from paper_2010_14298_gb300 import build
    path = build.build()
    lib = ctypes.CDLL(path)
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_status_strings_without_gpu():
    from paper_2010_14298_gb300 import fqt
    for code in range(7):
        assert fqt.status_string(code)
    assert fqt.status_string(4) == "non-finite input"


def test_argument_errors_are_synchronous_and_need_no_gpu():
    """Invalid arguments return FQT_EINVAL / FQT_EWORKSPACE before any launch."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    qs = fqt._QT()
    # null input
    st = lib.fqt_quantize_grad(None, 0, 16, 64, 0, 8, 0, 0, ctypes.byref(qs), None,
                               None, 0, None)
    assert st == 1
    # bad bits
    buf = ctypes.create_string_buffer(64)
    st = lib.fqt_quantize_act(ctypes.cast(buf, ctypes.c_void_p), 0, 4, 8, 9,
                              ctypes.byref(qs), None, 0, None)
    assert st == 1


def _aligned(n=1 << 16):
    """A 256-byte aligned host buffer standing in for a device pointer in
    calls that must fail validation before touching it."""
    raw = ctypes.create_string_buffer(n + 256)
    addr = (ctypes.addressof(raw) + 255) & ~255
    return raw, ctypes.c_void_p(addr)


def test_new_entry_points_validate_without_gpu():
    """The adaptive groups, the shift quantizer and the implicit im2col
    operand reject bad requests synchronously, before any CUDA call."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    raw, p = _aligned()
    q = fqt._QT()
    q.codes_f16 = p.value
    q.inv_s = p.value
    q.zero = p.value
    BHQ, SHIFT = 2, 3
    # adaptive BHQ (block 0) needs perm / gstart / gsize
    st = lib.fqt_quantize_grad(p, 0, 16, 64, BHQ, 5, 0, 0, ctypes.byref(q), None, p, 256,
                               None)
    assert st == 1
    # unknown kind
    assert lib.fqt_quantize_grad(p, 0, 16, 64, 7, 5, 0, 0, ctypes.byref(q), None, p, 256,
                                 None) == 1
    # the shift quantizer needs its grad_W operand arrays
    assert lib.fqt_quantize_grad(p, 0, 16, 64, SHIFT, 5, 0, 0, ctypes.byref(q), None, p, 256,
                                 None) == 1
    q.shift_f16 = p.value
    q.shift = p.value
    q.shift_col_sum = p.value
    q.shift_scale = p.value
    # ... and rows of 64 .. 1024 columns
    assert lib.fqt_quantize_grad(p, 0, 16, 72, SHIFT, 5, 0, 0, ctypes.byref(q), None, p, 256,
                                 None) == 2
    # the implicit im2col quantizer: row sums are not built, bad geometry fails
    qc = fqt._QT()
    qc.codes_f16 = p.value
    qc.inv_s = p.value
    qc.zero = p.value
    qc.col_sum = p.value
    qc.row_sum = p.value
    assert lib.fqt_quantize_act_conv(p, 0, 2, 8, 8, 64, 3, 3, 1, 8, ctypes.byref(qc), p, 256,
                                     None) == 2
    qc.row_sum = None
    assert lib.fqt_quantize_act_conv(p, 0, 2, 2, 2, 64, 5, 5, 0, 8, ctypes.byref(qc), p, 256,
                                     None) == 1  # 5x5 taps on a 2x2 image
    assert lib.fqt_quantize_act_conv(p, 0, 2, 8, 8, 60, 3, 3, 1, 8, ctypes.byref(qc), p, 256,
                                     None) == 2  # c % 8 != 0
    del raw


def test_adaptive_group_limits_without_gpu():
    """Adaptive BHQ groups (block 0): rows of 64, 128 or 256 columns and at
    most 2^20 rows (the radix sort's per-tile prefix); other requests are
    refused synchronously with FQT_EUNSUPPORTED."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    raw, p = _aligned()
    q = fqt._QT()
    for name in ("codes_f16", "inv_s", "zero", "row_sum", "hz", "hr", "perm", "gstart",
                 "gsize"):
        setattr(q, name, p.value)
    BHQ = 2
    assert lib.fqt_quantize_grad(p, 0, 64, 512, BHQ, 5, 0, 0, ctypes.byref(q), None, p, 256,
                                 None) == 2
    assert lib.fqt_quantize_grad(p, 0, (1 << 20) + 1, 64, BHQ, 5, 0, 0, ctypes.byref(q), None,
                                 p, 256, None) == 2
    # block sizes other than 0 or a power of two up to 128 are invalid
    assert lib.fqt_quantize_grad(p, 0, 64, 64, BHQ, 5, 24, 0, ctypes.byref(q), None, p, 256,
                                 None) == 1
    assert lib.fqt_quantize_grad(p, 0, 64, 64, BHQ, 5, 256, 0, ctypes.byref(q), None, p, 256,
                                 None) == 1
    del raw


def test_backward_shape_checks_without_gpu():
    """fqt_linear_backward refuses, before any launch: contraction widths
    that are not multiples of 16 or exceed the int32 epilogue bound
    (FQT_EUNSUPPORTED), mismatched operands and BHQ tensors without their
    lead rows or offsets (FQT_EINVAL), a misaligned workspace
    (FQT_EWORKSPACE)."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    raw, p = _aligned()

    def qt(rows, cols, kind=0, block=0, **fields):
        q = fqt._QT()
        q.rows, q.cols, q.bits, q.kind, q.block = rows, cols, 8, kind, block
        for name in ("codes_f16", "inv_s", "zero", "row_sum", "col_sum"):
            setattr(q, name, p.value)
        for k, v in fields.items():
            setattr(q, k, v)
        return q

    def run(q2, qw, ws=p):
        return lib.fqt_linear_backward(ctypes.byref(q2), None, None, ctypes.byref(qw), p, None,
                                       ws, 1 << 16, None)

    assert run(qt(256, 72), qt(72, 64)) == 2            # C % 16
    assert run(qt(256, 64), qt(64, 40)) == 2            # D % 16
    assert run(qt(256, 8208), qt(8208, 64)) == 2        # C above the int32 epilogue bound
    assert run(qt(256, 64), qt(128, 64)) == 1           # W~ rows != C
    assert run(qt(256, 64, kind=2, block=16), qt(64, 64)) == 1  # BHQ without lead / hz / hr
    assert run(qt(256, 64, kind=2, block=16, lead=p.value, hz=p.value), qt(64, 64)) == 1
    misaligned = ctypes.c_void_p(p.value + 64)
    assert run(qt(256, 64), qt(64, 64), ws=misaligned) == 6
    del raw


def test_fixed_scratch_and_wait_test_refusals_without_gpu():
    """fqt_grad_w_fixed_scratch refuses an implicit im2col operand
    (FQT_EUNSUPPORTED) and fqt_debug_wait_timeout a limit above 10 s or a
    misaligned workspace, all before any CUDA call."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    raw, p = _aligned()

    def qt(rows, cols, conv=None):
        q = fqt._QT()
        q.rows, q.cols, q.bits, q.kind = rows, cols, 8, 0
        for name in ("codes_f16", "inv_s", "zero", "col_sum"):
            setattr(q, name, p.value)
        if conv:
            q.conv = (ctypes.c_int32 * 8)(*conv)
        return q

    q1 = qt(2048, 64)
    qx = qt(2048, 576, conv=(2, 32, 32, 64, 3, 3, 1, 0))
    assert lib.fqt_grad_w_fixed_scratch(ctypes.byref(q1), ctypes.byref(qx), p, None) == 2
    assert lib.fqt_grad_w_fixed_scratch(ctypes.byref(qx), ctypes.byref(q1), p, None) == 2
    assert lib.fqt_debug_wait_timeout(p, 256, 10_000_000_001, None) == 1
    assert lib.fqt_debug_wait_timeout(ctypes.c_void_p(p.value + 16), 256, 1000, None) == 6
    assert lib.fqt_debug_wait_timeout(p, 128, 1000, None) == 6
    del raw


def test_sample_and_nhwc_refusals_without_gpu():
    """fqt_quantize_grad_samples and fqt_conv_grad_x_nhwc refuse bad requests
    before any CUDA call: rows that are not whole samples, BHQ samples, a
    5 x 5 kernel, per-row scales."""
    from paper_2010_14298_gb300 import fqt
    lib = fqt.load()
    raw, p = _aligned()
    q = fqt._QT()
    for name in ("codes_f16", "inv_s", "zero", "row_sum", "col_sum"):
        setattr(q, name, p.value)
    PSQ, BHQ = 1, 2
    assert lib.fqt_quantize_grad_samples(p, 0, 100, 64, 30, PSQ, 5, 0, ctypes.byref(q), None, p,
                                         1 << 16, None) == 1
    assert lib.fqt_quantize_grad_samples(p, 0, 100, 64, 10, BHQ, 5, 0, ctypes.byref(q), None, p,
                                         1 << 16, None) == 2
    assert lib.fqt_quantize_grad_samples(p, 0, 100, 72, 10, PSQ, 5, 0, ctypes.byref(q), None, p,
                                         1 << 16, None) == 2
    q2 = fqt._QT()
    q2.rows, q2.cols, q2.bits, q2.kind, q2.rows_per_sample = 2 * 8 * 8, 64, 5, PSQ, 64
    qw = fqt._QT()
    qw.rows, qw.cols, qw.bits, qw.kind = 64, 9 * 32, 8, 0
    for s in (q2, qw):
        for name in ("codes_f16", "inv_s", "zero", "row_sum", "col_sum"):
            setattr(s, name, p.value)
    out = p
    assert lib.fqt_conv_grad_x_nhwc(ctypes.byref(q2), ctypes.byref(qw), 2, 8, 8, 32, 5, 2, out, p,
                                     1 << 16, None) == 2
    q2.rows_per_sample = 1  # per-row scales do not factor out of the taps
    assert lib.fqt_conv_grad_x_nhwc(ctypes.byref(q2), ctypes.byref(qw), 2, 8, 8, 32, 3, 1, out, p,
                                     1 << 16, None) == 2
    q2.rows_per_sample = 64
    assert lib.fqt_conv_grad_x_nhwc(ctypes.byref(q2), ctypes.byref(qw), 2, 8, 8, 32, 3, 1, out, p,
                                     64, None) == 6  # workspace too small
    del raw
