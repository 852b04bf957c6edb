"""ctypes binding of the C ABI in include/fqt.h.

Argument marshalling only: every step of the hot path runs in the CUDA
library ``_lib/libfqt.so``.  PyTorch provides device memory and streams.
There is no CPU fallback: if the library is missing or no GPU is present the
calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass
from typing import Optional

import torch

from . import build as _build

PTQ, PSQ, BHQ, SHIFT = 0, 1, 2, 3
F32, BF16 = 0, 1
STATUS = {0: "FQT_OK", 1: "FQT_EINVAL", 2: "FQT_EUNSUPPORTED", 3: "FQT_ECUDA",
          4: "FQT_ENONFINITE", 5: "FQT_ETIMEOUT", 6: "FQT_EWORKSPACE"}

_lib = None
_lock = threading.Lock()


class FqtError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS.get(status, status)}")


class _QT(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("bits", ctypes.c_int32), ("kind", ctypes.c_int32),
                ("block", ctypes.c_int32), ("rows_per_sample", ctypes.c_int32),
                ("codes", ctypes.c_void_p), ("inv_s", ctypes.c_void_p),
                ("zero", ctypes.c_void_p), ("row_sum", ctypes.c_void_p),
                ("col_sum", ctypes.c_void_p), ("lead", ctypes.c_void_p),
                ("codes_f16", ctypes.c_void_p), ("hz", ctypes.c_void_p),
                ("hr", ctypes.c_void_p), ("perm", ctypes.c_void_p),
                ("gstart", ctypes.c_void_p), ("gsize", ctypes.c_void_p),
                ("shift_f16", ctypes.c_void_p), ("shift", ctypes.c_void_p),
                ("shift_col_sum", ctypes.c_void_p), ("shift_scale", ctypes.c_void_p),
                ("conv", ctypes.c_int32 * 8)]


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Loads libfqt.so (building it with nvcc when absent)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if not os.path.exists(path):
            if not build_if_missing:
                raise FileNotFoundError(f"{path} is not built")
            _build.build()
        lib = ctypes.CDLL(path)
        P, i64, u64, i32, sz = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_uint64,
                                ctypes.c_int, ctypes.c_size_t)
        QP = ctypes.POINTER(_QT)
        lib.fqt_workspace_size.argtypes = [i64, i64, i64]
        lib.fqt_workspace_size.restype = sz
        lib.fqt_debug_workspace_size.argtypes = [i64, i64, i64]
        lib.fqt_debug_workspace_size.restype = sz
        for name in ("fqt_quantize_act", "fqt_quantize_weight"):
            f = getattr(lib, name)
            f.argtypes = [P, i32, i64, i64, i32, QP, P, sz, P]
            f.restype = i32
        lib.fqt_quantize_grad.argtypes = [P, i32, i64, i64, i32, i32, i32, u64,
                                          QP, QP, P, sz, P]
        lib.fqt_quantize_grad.restype = i32
        lib.fqt_quantize_grad_samples.argtypes = [P, i32, i64, i64, i64, i32, i32, u64,
                                                  QP, QP, P, sz, P]
        lib.fqt_quantize_grad_samples.restype = i32
        lib.fqt_conv_grad_x_workspace_size.argtypes = [i64]
        lib.fqt_conv_grad_x_workspace_size.restype = sz
        lib.fqt_conv_grad_x_nhwc.argtypes = [QP, QP, i64, i64, i64, i64, i32, i32, P, P, sz, P]
        lib.fqt_conv_grad_x_nhwc.restype = i32
        lib.fqt_linear_backward.argtypes = [QP, QP, QP, QP, P, P, P, sz, P]
        lib.fqt_linear_backward.restype = i32
        lib.fqt_linear_forward.argtypes = [QP, QP, P, P, sz, P]
        lib.fqt_linear_forward.restype = i32
        lib.fqt_quantize_act_conv.argtypes = [P, i32, i64, i64, i64, i64, i32, i32, i32, i32,
                                              QP, P, sz, P]
        lib.fqt_quantize_act_conv.restype = i32
        lib.fqt_linear_forward.restype = i32
        lib.fqt_grad_w_fixed_scratch.argtypes = [QP, QP, P, P]
        lib.fqt_grad_w_fixed_scratch.restype = i32
        lib.fqt_sync_status.argtypes = [P, P]
        lib.fqt_sync_status.restype = i32
        lib.fqt_fixed_scratch_sync_status.argtypes = [P]
        lib.fqt_fixed_scratch_sync_status.restype = i32
        lib.fqt_debug_wait_timeout.argtypes = [P, sz, u64, P]
        lib.fqt_debug_wait_timeout.restype = i32
        lib.fqt_debug_mma_peak.argtypes = [i32, i64, ctypes.POINTER(ctypes.c_double), P, sz,
                                           P]
        lib.fqt_debug_mma_peak.restype = i32
        lib.fqt_debug_int_gemm.argtypes = [P, i32, i32, P, i32, i32, i64, i64,
                                           i64, P, P, sz, P]
        lib.fqt_debug_int_gemm.restype = i32
        lib.fqt_debug_int_gemm_u8.argtypes = [P, i32, P, i32, i64, i64, i64, P, P, sz, P]
        lib.fqt_debug_int_gemm_u8.restype = i32
        lib.fqt_status_string.argtypes = [i32]
        lib.fqt_status_string.restype = ctypes.c_char_p
        lib.fqt_last_cuda_error.argtypes = []
        lib.fqt_last_cuda_error.restype = ctypes.c_char_p
        _lib = lib
        return lib


def _check(st: int, what: str):
    if st != 0:
        if st == 3:
            what += " (" + load().fqt_last_cuda_error().decode() + ")"
        raise FqtError(st, what)


def _ptr(t: Optional[torch.Tensor]):
    return ctypes.c_void_p(t.data_ptr()) if t is not None else None


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported dtype {t.dtype}")


class Workspace:
    """Caller-owned device scratch (zero-filled once), see fqt_workspace_size."""

    def __init__(self, N: int, C: int, D: int, device="cuda"):
        self.nbytes = int(load().fqt_workspace_size(N, C, D))
        self.buf = torch.zeros(self.nbytes, dtype=torch.uint8, device=device)

    def ensure(self, N: int, C: int, D: int):
        need = int(load().fqt_workspace_size(N, C, D))
        if need > self.nbytes:
            self.nbytes = need
            self.buf = torch.zeros(need, dtype=torch.uint8, device=self.buf.device)
        return self

    @property
    def ptr(self):
        return ctypes.c_void_p(self.buf.data_ptr())


@dataclass
class QTensor:
    """A quantized matrix (the fqt_qtensor of include/fqt.h) held in torch tensors.

    ``codes`` holds the integer codes (uint8), ``codes16`` the same codes
    centred by 2^(b-1) as exact fp16 values (the tensor-core operand format);
    either may be None.  ``hz`` and ``hr`` (BHQ, block != 1) are the reflected
    per-row offsets the grad_X epilogue reads.  BHQ with block 0 takes the
    adaptive groups of App. D.5: rows are stored group by group, ``perm``
    maps a stored row to its row of dH, ``gstart`` holds the group starts
    (then N) and ``gsize`` every stored row's group size.  SHIFT (the
    per-sample power-of-two shift quantizer of Sec. 4.3) also carries
    ``shift`` (per row), ``shift16`` (the codes on the common scale, the
    grad_W operand), ``shift_col_sum`` and ``shift_scale`` (2^-4 / s, 0).
    """
    codes: Optional[torch.Tensor]
    inv_s: torch.Tensor
    zero: torch.Tensor
    row_sum: Optional[torch.Tensor]
    col_sum: Optional[torch.Tensor]
    lead: Optional[torch.Tensor]
    kind: int = PTQ
    bits: int = 8
    block: int = 0
    codes16: Optional[torch.Tensor] = None
    hz: Optional[torch.Tensor] = None
    hr: Optional[torch.Tensor] = None
    perm: Optional[torch.Tensor] = None
    gstart: Optional[torch.Tensor] = None
    gsize: Optional[torch.Tensor] = None
    shift16: Optional[torch.Tensor] = None
    shift: Optional[torch.Tensor] = None
    shift_col_sum: Optional[torch.Tensor] = None
    shift_scale: Optional[torch.Tensor] = None
    conv: Optional[tuple] = None   # implicit im2col operand: (n, h, w, c, kh, kw, pad, 0)
    rows_per_sample: int = 1       # rows of dH per sample (quantize_grad_samples)
    logical: Optional[tuple] = None  # (rows, cols) of that im2col matrix

    @property
    def shape(self):
        if self.logical is not None:
            return self.logical
        return (self.codes if self.codes is not None else self.codes16).shape

    @staticmethod
    def empty(rows: int, cols: int, kind: int, bits: int, block: int = 0,
              row_sum: bool = True, col_sum: bool = True, device="cuda",
              u8: bool = True, f16: bool = True):
        m = 1 if kind == PTQ else rows
        adaptive = kind == BHQ and block == 0
        nblk = (rows + block - 1) // block if kind == BHQ and not adaptive else 0
        offsets = kind == BHQ and block != 1 and row_sum
        i32 = lambda n: torch.empty(n, dtype=torch.int32, device=device)
        return QTensor(
            codes=(torch.empty((rows, cols), dtype=torch.uint8, device=device)
                   if u8 else None),
            codes16=(torch.empty((rows, cols), dtype=torch.float16, device=device)
                     if f16 else None),
            inv_s=torch.empty(m, dtype=torch.float32, device=device),
            zero=torch.empty(m, dtype=torch.float32, device=device),
            row_sum=(torch.empty(rows, dtype=torch.int32, device=device)
                     if row_sum else None),
            col_sum=(torch.empty(cols, dtype=torch.int32, device=device)
                     if col_sum else None),
            lead=i32(max(nblk, 1)) if kind == BHQ else None,
            kind=kind, bits=bits, block=block,
            hz=(torch.empty(rows, dtype=torch.float32, device=device)
                if offsets else None),
            hr=(torch.empty(rows, dtype=torch.float32, device=device)
                if offsets else None),
            perm=i32(max(rows, 1)) if adaptive else None,
            gstart=i32(rows + 1) if adaptive else None,
            gsize=i32(max(rows, 1)) if adaptive else None,
            shift16=(torch.empty((rows, cols), dtype=torch.float16, device=device)
                     if kind == SHIFT else None),
            shift=i32(max(rows, 1)) if kind == SHIFT else None,
            shift_col_sum=i32(cols) if kind == SHIFT else None,
            shift_scale=(torch.empty(2, dtype=torch.float32, device=device)
                         if kind == SHIFT else None))

    def c_struct(self) -> _QT:
        rows, cols = self.shape
        p = lambda t: t.data_ptr() if t is not None else None
        return _QT(rows, cols, self.bits, self.kind, self.block, self.rows_per_sample,
                   p(self.codes), self.inv_s.data_ptr(), self.zero.data_ptr(),
                   p(self.row_sum), p(self.col_sum), p(self.lead), p(self.codes16),
                   p(self.hz), p(self.hr), p(self.perm), p(self.gstart), p(self.gsize),
                   p(self.shift16), p(self.shift), p(self.shift_col_sum), p(self.shift_scale),
                   (ctypes.c_int32 * 8)(*(self.conv or (0,) * 8)))

    def codes_from_f16(self) -> torch.Tensor:
        """The uint8 codes recovered from the fp16 carriers."""
        off = 1 << (self.bits - 1)
        return (self.codes16.float() + off).round().to(torch.uint8)

    def to_numpy(self) -> dict:
        """Host copy in the oracle's dict layout."""
        codes = self.codes if self.codes is not None else self.codes_from_f16()
        d = dict(codes=codes.cpu().numpy(), inv_s=self.inv_s.cpu().numpy(),
                 zero=self.zero.cpu().numpy(), kind=self.kind, bits=self.bits,
                 block=self.block,
                 lead=(self.lead.cpu().numpy()
                       if self.kind == BHQ and self.block != 0 else None))
        if self.shift is not None:
            d["shift"] = self.shift.cpu().numpy()[:codes.shape[0]]
        if self.perm is not None:
            n = codes.shape[0]
            gs = self.gstart.cpu().numpy()
            d.update(perm=self.perm.cpu().numpy()[:n], gstart=gs,
                     gsize=self.gsize.cpu().numpy()[:n], G=int((gs[:n] < n).sum()))
        if self.row_sum is not None:
            d["row_sum"] = self.row_sum.cpu().numpy()
        if self.col_sum is not None:
            d["col_sum"] = self.col_sum.cpu().numpy()
        return d


def workspace_size(N: int, C: int, D: int) -> int:
    return int(load().fqt_workspace_size(N, C, D))


def _fwd(name, X, bits, ws, out, row_sum, col_sum, stream):
    lib = load()
    rows, cols = X.shape
    if out is None:
        out = QTensor.empty(rows, cols, PTQ, bits, 0, row_sum, col_sum, X.device)
    qs = out.c_struct()
    st = getattr(lib, name)(_ptr(X), _dtype_code(X), rows, cols, bits,
                            ctypes.byref(qs), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, name)
    out.kind, out.bits, out.block = PTQ, bits, 0
    return out


def quantize_act(X: torch.Tensor, bits: int = 8, ws: Workspace = None,
                 out: QTensor = None, row_sum: bool = False,
                 col_sum: bool = True, stream=None) -> QTensor:
    """X~ = Q_f(X): deterministic PTQ (Sec. 2.1, App. E)."""
    ws = ws or Workspace(*X.shape, 16, device=X.device)
    return _fwd("fqt_quantize_act", X.contiguous(), bits, ws, out, row_sum,
                col_sum, stream)


def quantize_act_conv(X: torch.Tensor, kh: int, kw: int, pad: int, bits: int = 8,
                      ws: Workspace = None, out: QTensor = None, u8: bool = False,
                      stream=None) -> QTensor:
    """X~ = Q_f(im2col(X)) for a stride-1 convolution, without forming the
    im2col matrix (Sec. 2.1, App. E): X is NHWC; the codes are stored NHWC
    and col_sum ends with the code of 0.0, the padding's code
    (fqt_quantize_act_conv)."""
    lib = load()
    X = X.contiguous()
    n, h, w, c = X.shape
    oh, ow = h + 2 * pad - kh + 1, w + 2 * pad - kw + 1
    dev = X.device
    ws = ws or Workspace(n * h * w, c, 16, device=dev)
    if out is None:
        out = QTensor(
            codes=(torch.empty((n * h * w, c), dtype=torch.uint8, device=dev) if u8 else None),
            codes16=torch.empty((n * h * w, c), dtype=torch.float16, device=dev),
            inv_s=torch.empty(1, dtype=torch.float32, device=dev),
            zero=torch.empty(1, dtype=torch.float32, device=dev),
            row_sum=None,
            col_sum=torch.empty(kh * kw * c + 1, dtype=torch.int32, device=dev),
            lead=None)
    out.logical = (n * oh * ow, kh * kw * c)
    qs = out.c_struct()
    st = lib.fqt_quantize_act_conv(_ptr(X), _dtype_code(X), n, h, w, c, kh, kw, pad, bits,
                                   ctypes.byref(qs), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "fqt_quantize_act_conv")
    out.kind, out.bits, out.block = PTQ, bits, 0
    out.conv = tuple(qs.conv)
    return out


def quantize_weight(W: torch.Tensor, bits: int = 8, ws: Workspace = None,
                    out: QTensor = None, row_sum: bool = False,
                    col_sum: bool = True, stream=None) -> QTensor:
    """W~ = Q_theta(W): deterministic PTQ (Sec. 2.1, App. E)."""
    ws = ws or Workspace(*W.shape, 16, device=W.device)
    return _fwd("fqt_quantize_weight", W.contiguous(), bits, ws, out, row_sum,
                col_sum, stream)


def quantize_grad(dH: torch.Tensor, kind: int, bits: int, block: int = 0,
                  seed: int = 0, with_b1: bool = True, ws: Workspace = None,
                  q_b2: QTensor = None, q_b1: QTensor = None,
                  b2_col_sum: bool = False, stream=None):
    """(Q_b2(dH), Q_b1(dH)) with stochastic rounding (Sec. 3.3, 4.1, 4.2, App. E)."""
    lib = load()
    dH = dH.contiguous()
    N, C = dH.shape
    ws = ws or Workspace(N, C, 16, device=dH.device)
    if q_b2 is None:
        q_b2 = QTensor.empty(N, C, kind, bits, block if kind == BHQ else 0,
                             True, b2_col_sum or not with_b1, dH.device)
    if with_b1 and q_b1 is None:
        q_b1 = QTensor.empty(N, C, PTQ, 8, 0, False, True, dH.device)
    s2 = q_b2.c_struct()
    s1 = q_b1.c_struct() if with_b1 else None
    st = lib.fqt_quantize_grad(_ptr(dH), _dtype_code(dH), N, C, kind, bits,
                               block if kind == BHQ else 0,
                               ctypes.c_uint64(seed & (2 ** 64 - 1)),
                               ctypes.byref(s2),
                               ctypes.byref(s1) if s1 is not None else None,
                               ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "fqt_quantize_grad")
    q_b2.kind, q_b2.bits, q_b2.block = kind, bits, block if kind == BHQ else 0
    if with_b1:
        q_b1.kind, q_b1.bits, q_b1.block = PTQ, 8, 0
    return q_b2, (q_b1 if with_b1 else None)


def quantize_grad_samples(dH: torch.Tensor, rows_per_sample: int, kind: int, bits: int,
                          seed: int = 0, with_b1: bool = True, ws: Workspace = None,
                          q_b2: QTensor = None, q_b1: QTensor = None, stream=None):
    """(Q_b2, Q_b1) with one sample per `rows_per_sample` rows of dH (an
    image's output pixels; Sec. 4.1): fqt_quantize_grad_samples."""
    lib = load()
    dH = dH.contiguous()
    N, C = dH.shape
    ws = ws or Workspace(N, C, 16, device=dH.device)
    if q_b2 is None:
        q_b2 = QTensor.empty(N, C, kind if kind != PTQ else PTQ, bits, 0, True,
                             not with_b1, dH.device)
    if with_b1 and q_b1 is None:
        q_b1 = QTensor.empty(N, C, PTQ, 8, 0, False, True, dH.device)
    s2 = q_b2.c_struct()
    s1 = q_b1.c_struct() if with_b1 else None
    st = lib.fqt_quantize_grad_samples(_ptr(dH), _dtype_code(dH), N, C, rows_per_sample, kind,
                                       bits, ctypes.c_uint64(seed & (2 ** 64 - 1)),
                                       ctypes.byref(s2),
                                       ctypes.byref(s1) if s1 is not None else None,
                                       ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "fqt_quantize_grad_samples")
    q_b2.kind, q_b2.bits, q_b2.block = kind, bits, 0
    q_b2.rows_per_sample = rows_per_sample
    if with_b1:
        q_b1.kind, q_b1.bits, q_b1.block = PTQ, 8, 0
    return q_b2, (q_b1 if with_b1 else None)


def linear_forward(qx: QTensor, qw: QTensor, ws: Workspace = None, out: torch.Tensor = None,
                   stream=None) -> torch.Tensor:
    """H = X~ W~^T (Sec. 2.1): the quantized forward of the layer (N x C fp32).
    qx and qw need codes16 and row_sum (quantize_act / quantize_weight with
    row_sum=True)."""
    lib = load()
    N, D = qx.shape
    C = qw.shape[0]
    dev = qx.inv_s.device
    ws = ws or Workspace(N, C, D, device=dev)
    if out is None:
        out = torch.empty((N, C), dtype=torch.float32, device=dev)
    sx, sw = qx.c_struct(), qw.c_struct()
    st = lib.fqt_linear_forward(ctypes.byref(sx), ctypes.byref(sw), _ptr(out), ws.ptr,
                                ws.nbytes, _stream(stream))
    _check(st, "fqt_linear_forward")
    return out


def linear_backward(q_b2: QTensor, q_b1: Optional[QTensor], qx: QTensor,
                    qw: QTensor, grad_x: bool = True, grad_w: bool = True,
                    ws: Workspace = None, out_x: torch.Tensor = None,
                    out_w: torch.Tensor = None, stream=None):
    """grad_X = Q_b2(dH) W~ and grad_W = Q_b1(dH)^T X~ (Eq. 6, App. E)."""
    lib = load()
    N, C = q_b2.shape
    D = qx.shape[1] if qx is not None else qw.shape[1]
    dev = q_b2.inv_s.device
    ws = (ws or Workspace(N, C, D, device=dev)).ensure(N, C, D)
    gx = gw = None
    if grad_x:
        gx = out_x if out_x is not None else torch.empty((N, D), dtype=torch.float32,
                                                         device=dev)
    if grad_w:
        gw = out_w if out_w is not None else torch.empty((C, D), dtype=torch.float32,
                                                         device=dev)
    s2 = q_b2.c_struct()
    s1 = q_b1.c_struct() if q_b1 is not None else None
    sx = qx.c_struct() if qx is not None else None
    sw = qw.c_struct() if qw is not None else None
    st = lib.fqt_linear_backward(ctypes.byref(s2),
                                 ctypes.byref(s1) if s1 is not None else None,
                                 ctypes.byref(sx) if sx is not None else None,
                                 ctypes.byref(sw) if sw is not None else None,
                                 _ptr(gx), _ptr(gw), ws.ptr, ws.nbytes,
                                 _stream(stream))
    _check(st, "fqt_linear_backward")
    return gx, gw


def conv_grad_x_nhwc(q_b2: QTensor, qw: QTensor, n: int, h: int, w: int, cin: int,
                     k: int = 3, pad: int = 1, ws: Workspace = None,
                     out: torch.Tensor = None, stream=None) -> torch.Tensor:
    """grad_X of a stride-1 conv in NHWC with col2im fused into the contraction
    (fqt_conv_grad_x_nhwc); q_b2 PTQ or per-image PSQ (quantize_grad_samples
    with rows_per_sample = h w)."""
    lib = load()
    dev = q_b2.inv_s.device
    if out is None:
        out = torch.empty((n, h, w, cin), dtype=torch.float32, device=dev)
    need = int(lib.fqt_conv_grad_x_workspace_size(cin))
    if ws is None or ws.nbytes < need:
        ws = Workspace(1, 16, 16, device=dev)
        ws.nbytes = need
        ws.buf = torch.zeros(need, dtype=torch.uint8, device=dev)
    s2, sw = q_b2.c_struct(), qw.c_struct()
    st = lib.fqt_conv_grad_x_nhwc(ctypes.byref(s2), ctypes.byref(sw), n, h, w, cin, k, pad,
                                  _ptr(out), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "fqt_conv_grad_x_nhwc")
    return out


def grad_w_fixed_scratch(q_b1: QTensor, qx: QTensor, out: torch.Tensor = None,
                         stream=None) -> torch.Tensor:
    """grad_W through fqt_grad_w_fixed_scratch: no workspace, the library's
    fixed scratch array holds the split-K partials (for callers that cannot
    allocate device memory at this point)."""
    lib = load()
    C, D = q_b1.shape[1], qx.shape[1]
    if out is None:
        out = torch.empty((C, D), dtype=torch.float32, device=q_b1.inv_s.device)
    s1, sx = q_b1.c_struct(), qx.c_struct()
    st = lib.fqt_grad_w_fixed_scratch(ctypes.byref(s1), ctypes.byref(sx), _ptr(out),
                                      _stream(stream))
    _check(st, "fqt_grad_w_fixed_scratch")
    return out


def debug_int_gemm(A: torch.Tensor, a_kmajor: bool, a_bits: int, B: torch.Tensor,
                   b_kmajor: bool, b_bits: int, M: int, N: int, K: int,
                   ws: Workspace = None, stream=None) -> torch.Tensor:
    """Exact sum_k (A_ik - 2^(a-1))(B_kj - 2^(b-1)) as int64 (M x N)."""
    lib = load()
    out = torch.empty((M, N), dtype=torch.int64, device=A.device)
    need = int(lib.fqt_debug_workspace_size(M, N, K))
    if ws is None or ws.nbytes < need:
        ws = Workspace(1, 16, 16, device=A.device)
        ws.nbytes = need
        ws.buf = torch.zeros(need, dtype=torch.uint8, device=A.device)
    st = lib.fqt_debug_int_gemm(_ptr(A), int(a_kmajor), a_bits, _ptr(B),
                                int(b_kmajor), b_bits, M, N, K, _ptr(out), ws.ptr,
                                ws.nbytes, _stream(stream))
    _check(st, "fqt_debug_int_gemm")
    return out


def debug_int_gemm_u8(A: torch.Tensor, a_bits: int, B: torch.Tensor, b_bits: int, M: int,
                      N: int, K: int, ws: Workspace = None, stream=None) -> torch.Tensor:
    """debug_int_gemm with both operands MN-major bytes (A: K x M, B: K x N),
    widened to fp16 carriers on chip (grad_W's byte-operand path)."""
    lib = load()
    out = torch.empty((M, N), dtype=torch.int64, device=A.device)
    need = int(lib.fqt_debug_workspace_size(M, N, K))
    if ws is None or ws.nbytes < need:
        ws = Workspace(1, 16, 16, device=A.device)
        ws.nbytes = need
        ws.buf = torch.zeros(need, dtype=torch.uint8, device=A.device)
    st = lib.fqt_debug_int_gemm_u8(_ptr(A), a_bits, _ptr(B), b_bits, M, N, K, _ptr(out),
                                   ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "fqt_debug_int_gemm_u8")
    return out


def sync_status(ws: Workspace, stream=None) -> int:
    """Synchronises and returns (then clears) the device-side status word."""
    return int(load().fqt_sync_status(ws.ptr, _stream(stream)))


def fixed_scratch_sync_status(stream=None) -> int:
    """Synchronises and returns (then clears) the status word of the fixed
    array behind grad_w_fixed_scratch."""
    return int(load().fqt_fixed_scratch_sync_status(_stream(stream)))


def debug_wait_timeout(limit_ns: int, ws: Optional[Workspace] = None, stream=None):
    """Enqueues a bounded wait that is made to run out after limit_ns; its
    FQT_ETIMEOUT lands in ws (or, with ws None, the fixed array's word)."""
    lib = load()
    st = lib.fqt_debug_wait_timeout(ws.ptr if ws is not None else None,
                                    ws.nbytes if ws is not None else 0,
                                    ctypes.c_uint64(limit_ns), _stream(stream))
    _check(st, "fqt_debug_wait_timeout")


def debug_mma_peak(kind: int, iters: int, ws: Workspace, stream=None) -> float:
    """Enqueues the rate kernel of `kind` (0 tcgen05 f16, 1 tcgen05 e4m3,
    2 mma.sync u8 x s8); returns the operations it performs."""
    ops = ctypes.c_double(0.0)
    _check(load().fqt_debug_mma_peak(kind, iters, ctypes.byref(ops), ws.ptr, ws.nbytes,
                                     _stream(stream)), "fqt_debug_mma_peak")
    return ops.value


def status_string(code: int) -> str:
    return load().fqt_status_string(code).decode()
