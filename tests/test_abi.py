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
