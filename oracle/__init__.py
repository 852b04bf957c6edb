"""CPU oracle for the FQT quantized backward pass (arXiv 2010.14298).

TEST INFRASTRUCTURE ONLY.  Only the test suite, ``__graft_entry__.smoke()``
and the CPU-baseline / reference leg of ``bench.py`` may import this package.
The CUDA library never calls it, and it shares no code with that library:
the arithmetic lives in ``fqt_oracle.c`` (plain C, one IEEE rounding per
operation, no FMA contraction) and in the plain loops here.

Every function cites the passage of the paper it restates:

* ``quantize_grad``  -- PTQ (Sec. 3.3), PSQ (Sec. 4.1), BHQ (Sec. 4.2, App. D.4)
* ``bhq_grouping``   -- the adaptive BHQ groups of App. D.5 (block = 0)
* SHIFT quantizer   -- per-tensor range, per-sample power-of-two shifts (Sec. 4.3)
* ``grad_w_shifted`` -- grad_W with the shifted integer accumulators of Sec. 4.3
* ``quantize_fwd``   -- deterministic 8-bit PTQ of X and W (Sec. 2.1, App. E)
* ``dequant``        -- Eq. 9: Q(dH) = S^-1 (codes + z' 1^T)
* ``grad_x``/``grad_w`` -- Eq. 6 with the bifurcation of App. E
* ``int_gemm``       -- the exact integer contraction the low-bit kernels do
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "fqt_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libfqt_oracle.so")
_lib = None
_lock = threading.Lock()

PTQ, PSQ, BHQ, SHIFT = 0, 1, 2, 3
STREAM_B2, STREAM_B1 = 0, 1


def build(force: bool = False) -> str:
    """Compile fqt_oracle.c into oracle/_build/libfqt_oracle.so with gcc."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c11", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i64, u64, u32, i32 = (ctypes.c_int64, ctypes.c_uint64, ctypes.c_uint32,
                              ctypes.c_int)
        lib.orc_philox4x32_10.argtypes = [P, P, P]
        lib.orc_philox4x32_10.restype = None
        lib.orc_u16.argtypes = [u64, u32, u64]
        lib.orc_u16.restype = u32
        lib.orc_sr.argtypes = [ctypes.c_float, u32, u32]
        lib.orc_sr.restype = u32
        lib.orc_sr_moments.argtypes = [ctypes.c_float, u32, P, P]
        lib.orc_sr_moments.restype = None
        lib.orc_range.argtypes = [P, i64, P, P]
        lib.orc_range.restype = i64
        lib.orc_quantize_grad.argtypes = [P, i64, i64, i32, i32, i32, u64, u32,
                                          P, P, P, P, P]
        lib.orc_quantize_grad.restype = i64
        lib.orc_quant_det.argtypes = [P, i64, i64, i32, P, P, P]
        lib.orc_quant_det.restype = i64
        lib.orc_householder.argtypes = [i32, i32, P]
        lib.orc_householder.restype = None
        lib.orc_bhq_scales.argtypes = [ctypes.c_double, ctypes.c_double, i32,
                                       u32, P, P]
        lib.orc_bhq_scales.restype = None
        lib.orc_dequant.argtypes = [P, i64, i64, i32, i32, P, P, P, P]
        lib.orc_dequant.restype = None
        lib.orc_dequant_f64.argtypes = [P, i64, i64, i32, i32, P, P, P, P]
        lib.orc_dequant_f64.restype = None
        lib.orc_int_gemm.argtypes = [P, i32, P, i32, i64, i64, i64, i32, i32, P]
        lib.orc_int_gemm.restype = None
        lib.orc_matmul_f64.argtypes = [P, i32, P, i64, i64, i64, P]
        lib.orc_matmul_f64.restype = None
        lib.orc_bhq_grouping.argtypes = [P, i64, i64, P, P, P, P, P]
        lib.orc_bhq_grouping.restype = i64
        lib.orc_quant_bhq_groups.argtypes = [P, i64, i64, i32, P, P, i64, u64,
                                             u32, P, P, P, P]
        lib.orc_quant_bhq_groups.restype = i64
        lib.orc_dequant_groups_f64.argtypes = [P, i64, i64, P, i64, P, P, P]
        lib.orc_dequant_groups_f64.restype = None
        lib.orc_col2im_nhwc.argtypes = [P, i64, i64, i64, i64, i32, i32, i32, i32, P]
        lib.orc_col2im_nhwc.restype = None
        _lib = lib
        return lib


def _ptr(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data) if a is not None else None


def _f32(x) -> np.ndarray:
    """fp32 C-contiguous copy of x (bf16 sources arrive already widened)."""
    return np.ascontiguousarray(np.asarray(x, dtype=np.float32))


class OracleError(RuntimeError):
    pass


# --------------------------------------------------------------------------
# Random numbers and stochastic rounding (Sec. 3.3 / App. D)
# --------------------------------------------------------------------------
def philox4x32_10(ctr, key) -> tuple:
    """One Philox4x32-10 block (Salmon et al., SC'11)."""
    lib = _load()
    c = np.asarray(ctr, dtype=np.uint32)
    k = np.asarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib.orc_philox4x32_10(_ptr(c), _ptr(k), _ptr(out))
    return tuple(int(x) for x in out)


def u16(seed: int, stream: int, idx: int) -> int:
    return int(_load().orc_u16(seed, stream, idx))


def sr(v: float, u: int, B: int) -> int:
    """SR(v) for one fixed uniform u (Sec. 3.3)."""
    return int(_load().orc_sr(float(v), int(u), int(B)))


def sr_moments(v: float, B: int) -> tuple:
    """Exact mean / variance of SR(v) by enumeration of every 16-bit uniform."""
    lib = _load()
    m = np.zeros(1)
    var = np.zeros(1)
    lib.orc_sr_moments(float(v), int(B), _ptr(m), _ptr(var))
    return float(m[0]), float(var[0])


# --------------------------------------------------------------------------
# Quantizers
# --------------------------------------------------------------------------
def quantize_grad(dH, kind: int, bits: int, block: int = 0, seed: int = 0,
                  stream: int = STREAM_B2, want_v: bool = False) -> dict:
    """Gradient quantizer Q_b: PTQ (Sec. 3.3), PSQ (Sec. 4.1), BHQ (Sec. 4.2).

    Returns codes (uint8, N x C), inv_s and zero (1 entry for PTQ, N otherwise),
    lead (BHQ: lead row of each block) and, with want_v, the pre-rounding
    values v that SR acts on.  SHIFT (kind 3) is the per-tensor-range,
    per-sample-shift quantizer of Sec. 4.3 (reading R9 of fqt_oracle.c); its
    dict carries ``shift`` (per row) instead of lead.  BHQ with block = 0 takes the adaptive groups
    of App. D.5 (``bhq_grouping``): codes, inv_s, zero and v are then in the
    grouped (stored) order, row k holding row perm[k] of dH, and the dict
    also carries perm, gstart, gsize and G.
    """
    h = _f32(dH)
    n, c = h.shape
    if kind == BHQ and block < 0:
        raise OracleError("BHQ needs block >= 0 (0 = adaptive groups)")
    if kind == BHQ and block == 0:
        return _quantize_bhq_adaptive(h, bits, seed, stream, want_v)
    codes = np.zeros((n, c), dtype=np.uint8)
    m = 1 if kind == PTQ else n
    inv_s = np.zeros(m, dtype=np.float32)
    zero = np.zeros(m, dtype=np.float32)
    nblk = (n + block - 1) // block if kind == BHQ else 0
    # BHQ: lead row of each block; SHIFT: the shift of each row
    lead = np.zeros(max(n if kind == SHIFT else nblk, 1), dtype=np.int32)
    v = np.zeros((n, c), dtype=np.float32) if want_v else None
    bad = _load().orc_quantize_grad(_ptr(h), n, c, kind, bits,
                                    block if kind == BHQ else 0, seed, stream,
                                    _ptr(codes), _ptr(inv_s), _ptr(zero),
                                    _ptr(lead), _ptr(v))
    if bad:
        raise OracleError(f"{bad} non-finite gradient entries")
    out = dict(codes=codes, inv_s=inv_s, zero=zero, kind=kind, bits=bits,
               block=block if kind == BHQ else 0,
               lead=lead[:nblk] if kind == BHQ else None)
    if kind == SHIFT:
        out["shift"] = lead[:n].copy()
    if want_v:
        out["v"] = v
    return out


def shifted_codes(q: dict) -> np.ndarray:
    """Integer codes of the shift quantizer on the common scale 1 / (16 s)
    (Sec. 4.3): a_ic = 2^(4 - shift_i) (code_ic - 2^(b-1)), exact in int64."""
    z0 = 1 << (q["bits"] - 1)
    sh = np.asarray(q["shift"], dtype=np.int64)
    return (np.asarray(q["codes"], dtype=np.int64) - z0) << (4 - sh)[:, None]


def grad_w_shifted(q: dict, q_x: dict) -> np.ndarray:
    """grad_W = Q(dH)^T X~ for the shift quantizer, as Sec. 4.3 describes the
    hardware form: every sample's integer products are shifted by its
    2^(4 - shift_i) before the sum over samples (exact int64), and one scale
    1 / (16 s) is applied at the end.  X~ = inv_sx (codes_x + zero_x)."""
    a = shifted_codes(q)                                   # N x C, int64
    cx = np.asarray(q_x["codes"], dtype=np.int64)          # N x D
    P = a.T @ cx                                           # exact
    colsum_a = a.sum(axis=0)                               # C
    inv16s = float(np.float64(q["inv_s"][0]) * 2.0 ** (int(q["shift"][0]) - 4)) \
        if len(q["shift"]) else 0.0
    ix, zx = float(q_x["inv_s"][0]), float(q_x["zero"][0])
    return inv16s * ix * (P.astype(np.float64) + zx * colsum_a[:, None].astype(np.float64))


def bhq_grouping(dH, want_v: bool = False) -> dict:
    """Adaptive BHQ grouping of App. D.5 (reading R8 of fqt_oracle.c).

    Rows sorted by M_i = ||h_i||_inf (descending, ties by index); for every
    group count G the estimate V(G) of App. D.4's bound with the paper's
    group sizes (N - G) M_i / sum M; G = argmin V; integer sizes by
    cumulative rounding.  Returns perm (stored row -> dH row), gstart (G + 1
    group starts, then N repeated up to N + 1 entries), gsize (per stored
    row), G and, with want_v, V (V[G - 1] = V(G), N - 1 entries).
    """
    h = _f32(dH)
    n, c = h.shape
    perm = np.zeros(max(n, 1), dtype=np.int32)
    gstart = np.zeros(n + 1, dtype=np.int32)
    gsize = np.zeros(max(n, 1), dtype=np.int32)
    G = np.zeros(1, dtype=np.int64)
    V = np.zeros(max(n - 1, 1)) if want_v else None
    bad = _load().orc_bhq_grouping(_ptr(h), n, c, _ptr(perm), _ptr(gstart),
                                   _ptr(gsize), _ptr(G), _ptr(V))
    if bad:
        raise OracleError(f"{bad} non-finite gradient entries")
    out = dict(perm=perm[:n], gstart=gstart, gsize=gsize[:n], G=int(G[0]))
    if want_v:
        out["V"] = V[:max(n - 1, 0)]
    return out


def _quantize_bhq_adaptive(h, bits, seed, stream, want_v):
    n, c = h.shape
    grp = bhq_grouping(h)
    codes = np.zeros((n, c), dtype=np.uint8)
    inv_s = np.zeros(n, dtype=np.float32)
    zero = np.zeros(n, dtype=np.float32)
    v = np.zeros((n, c), dtype=np.float32) if want_v else None
    perm = np.ascontiguousarray(grp["perm"], dtype=np.int32)
    gstart = np.ascontiguousarray(grp["gstart"], dtype=np.int32)
    bad = _load().orc_quant_bhq_groups(_ptr(h), n, c, bits, _ptr(perm),
                                       _ptr(gstart), grp["G"], seed, stream,
                                       _ptr(codes), _ptr(inv_s), _ptr(zero),
                                       _ptr(v))
    if bad:
        raise OracleError(f"{bad} non-finite gradient entries")
    out = dict(codes=codes, inv_s=inv_s, zero=zero, kind=BHQ, bits=bits,
               block=0, lead=None, **grp)
    if want_v:
        out["v"] = v
    return out


def quantize_fwd(X, bits: int = 8) -> dict:
    """Deterministic PTQ of a forward operand, Q_f / Q_theta (Sec. 2.1, App. E)."""
    x = _f32(X)
    n, c = x.shape
    codes = np.zeros((n, c), dtype=np.uint8)
    inv_s = np.zeros(1, dtype=np.float32)
    zero = np.zeros(1, dtype=np.float32)
    bad = _load().orc_quant_det(_ptr(x), n, c, bits, _ptr(codes), _ptr(inv_s),
                                _ptr(zero))
    if bad:
        raise OracleError(f"{bad} non-finite entries")
    return dict(codes=codes, inv_s=inv_s, zero=zero, kind=PTQ, bits=bits,
                block=0, lead=None)


def householder(nb: int, p: int) -> np.ndarray:
    """Q = I - 2 n n^T / ||n||^2, n = 1/sqrt(N) 1 - e_p (Sec. 4.2)."""
    Q = np.zeros((nb, nb))
    _load().orc_householder(nb, p, _ptr(Q))
    return Q


def bhq_scales(lambda1: float, lambda2: float, nb: int, B: int) -> tuple:
    """s1, s2 of App. D.4 for one group of nb rows."""
    s1 = np.zeros(1)
    s2 = np.zeros(1)
    _load().orc_bhq_scales(float(lambda1), float(lambda2), nb, B, _ptr(s1),
                           _ptr(s2))
    return float(s1[0]), float(s2[0])


def dequant(q: dict, codes=None) -> np.ndarray:
    """The value the encoding represents, Eq. 9: diag(inv_s) Q_blk (codes + z').

    ``codes`` may be given as floats (e.g. expected codes); the map is affine
    in them, so dequant(E[codes]) = E[dequant(codes)].  For the adaptive BHQ
    groups (block = 0) the codes are in the stored order and the result is
    returned in dH's row order (row perm[k] <- stored row k).
    """
    src = q["codes"] if codes is None else codes
    lib = _load()
    if q["kind"] == BHQ and q.get("block", 0) == 0:
        cd = np.ascontiguousarray(src, dtype=np.float64)
        n, c = cd.shape
        stored = np.zeros((n, c))
        lib.orc_dequant_groups_f64(
            _ptr(cd), n, c, _ptr(np.ascontiguousarray(q["gstart"], dtype=np.int32)),
            q["G"], _ptr(np.ascontiguousarray(q["inv_s"], dtype=np.float32)),
            _ptr(np.ascontiguousarray(q["zero"], dtype=np.float32)), _ptr(stored))
        out = np.zeros((n, c))
        out[np.asarray(q["perm"], dtype=np.int64)] = stored
        return out
    if np.asarray(src).dtype == np.uint8:
        cd = np.ascontiguousarray(src, dtype=np.uint8)
        fn = lib.orc_dequant
    else:
        cd = np.ascontiguousarray(src, dtype=np.float64)
        fn = lib.orc_dequant_f64
    n, c = cd.shape
    out = np.zeros((n, c))
    inv_s = np.ascontiguousarray(q["inv_s"], dtype=np.float32)
    zero = np.ascontiguousarray(q["zero"], dtype=np.float32)
    lead = (np.ascontiguousarray(q["lead"], dtype=np.int32)
            if q.get("lead") is not None else np.zeros(1, dtype=np.int32))
    fn(_ptr(cd), n, c, q["kind"], max(q.get("block", 0), 1), _ptr(inv_s),
       _ptr(zero), _ptr(lead), _ptr(out))
    return out


# --------------------------------------------------------------------------
# Contractions (Eq. 6, App. E)
# --------------------------------------------------------------------------
def int_gemm(A, a_kmajor: bool, Bm, b_kmajor: bool, M: int, N: int, K: int,
             oa: int, ob: int) -> np.ndarray:
    """P_ij = sum_k (A_ik - oa)(B_kj - ob), exact in int64."""
    a = np.ascontiguousarray(A, dtype=np.uint8)
    b = np.ascontiguousarray(Bm, dtype=np.uint8)
    out = np.zeros((M, N), dtype=np.int64)
    _load().orc_int_gemm(_ptr(a), int(a_kmajor), _ptr(b), int(b_kmajor), M, N,
                         K, oa, ob, _ptr(out))
    return out


def matmul(A: np.ndarray, Bm: np.ndarray, a_trans: bool = False) -> np.ndarray:
    """Plain double product op(A) @ Bm with op(A) = A or A^T."""
    a = np.ascontiguousarray(A, dtype=np.float64)
    b = np.ascontiguousarray(Bm, dtype=np.float64)
    K, N = b.shape
    M = a.shape[1] if a_trans else a.shape[0]
    out = np.zeros((M, N))
    _load().orc_matmul_f64(_ptr(a), int(a_trans), _ptr(b), M, K, N, _ptr(out))
    return out


def grad_x(q_b2: dict, q_w: dict, codes_b2=None) -> np.ndarray:
    """grad_X = Q_b2(dH) W~ (Eq. 6 in the N x C, C x D layout; App. E)."""
    return matmul(dequant(q_b2, codes_b2), dequant(q_w))


def grad_w(q_b1: dict, q_x: dict, codes_b1=None) -> np.ndarray:
    """grad_W = Q_b1(dH)^T X~ (C x D; the transpose of Eq. 6's D x C form)."""
    return matmul(dequant(q_b1, codes_b1), dequant(q_x), a_trans=True)


# --------------------------------------------------------------------------
# Per-image samples and col2im (a conv layer as a linear layer on im2col rows,
# Sec. 2.1; a "sample" is one input's gradient, Sec. 4.1)
# --------------------------------------------------------------------------
def quantize_grad_samples(dH, rows_per_sample: int, kind: int, bits: int, block: int = 0,
                          seed: int = 0, stream: int = STREAM_B2, want_v: bool = False) -> dict:
    """Q_b2 with one sample per group of `rows_per_sample` consecutive rows of
    dH (an image's H W output pixels of a conv layer): the quantizer of the
    given kind applied to the (N / R) x (R C) matrix whose rows are the
    images' whole gradients.  The flat index of every entry, and so its SR
    uniform, is that of dH.  The dict is the quantizer's on that matrix
    (codes, inv_s, zero, lead, v reshaped to N x C) with ``rows_per_sample``
    set; ``inv_s_rows`` / ``zero_rows`` repeat the per-sample values for each
    row (PTQ keeps its single entry)."""
    h = _f32(dH)
    n, c = h.shape
    R = int(rows_per_sample)
    if R < 1 or n % R:
        raise OracleError("rows_per_sample must divide the rows")
    q = quantize_grad(h.reshape(n // R, R * c), kind, bits, block, seed, stream, want_v)
    q["codes"] = q["codes"].reshape(n, c)
    if want_v:
        q["v"] = q["v"].reshape(n, c)
    q["rows_per_sample"] = R
    if kind == PTQ:
        q["inv_s_rows"], q["zero_rows"] = q["inv_s"], q["zero"]
    else:
        q["inv_s_rows"] = np.repeat(q["inv_s"], R)
        q["zero_rows"] = np.repeat(q["zero"], R)
    return q


def dequant_samples(q: dict) -> np.ndarray:
    """The value of a per-sample quantized dH (N x C): Eq. 9 on the
    (N / R) x (R C) matrix of samples, read back as N x C."""
    R = q["rows_per_sample"]
    n, c = q["codes"].shape
    view = dict(q)
    view["codes"] = q["codes"].reshape(n // R, R * c)
    return dequant(view).reshape(n, c)


def col2im_nhwc(G, n: int, h: int, w: int, c: int, kh: int, kw: int, stride: int = 1,
                pad: int = 0) -> np.ndarray:
    """NHWC sum of an im2col-space gradient (the adjoint of im2col)."""
    g = np.ascontiguousarray(G, dtype=np.float64)
    oh = (h + 2 * pad - kh) // stride + 1
    ow = (w + 2 * pad - kw) // stride + 1
    if g.shape != (n * oh * ow, kh * kw * c):
        raise OracleError("G has the wrong shape for this geometry")
    out = np.zeros((n, h, w, c))
    _load().orc_col2im_nhwc(_ptr(g), n, h, w, c, kh, kw, stride, pad, _ptr(out))
    return out


def grad_x_nhwc(q_b2: dict, q_w: dict, n: int, h: int, w: int, cin: int, k: int,
                pad: int) -> np.ndarray:
    """grad_X of a stride-1 k x k conv in NHWC: col2im of Q_b2(dH) W~ (Eq. 6),
    Q_b2 per row, per sample (``rows_per_sample``) or per tensor."""
    deq = dequant_samples(q_b2) if "rows_per_sample" in q_b2 else dequant(q_b2)
    return col2im_nhwc(matmul(deq, dequant(q_w)), n, h, w, cin, k, k, 1, pad)


def linear_backward(dH, X, W, kind: int, bits: int, block: int, seed: int,
                    reuse_b2: bool = False) -> dict:
    """One FQT backward of a linear layer (Eq. 6 with App. E's bifurcation):
    Q_b2 (kind, bits) feeds grad_X, 8-bit stochastic PTQ Q_b1 feeds grad_W,
    X~ and W~ are the deterministic 8-bit forward codes."""
    q_x = quantize_fwd(X, 8)
    q_w = quantize_fwd(W, 8)
    q_b2 = quantize_grad(dH, kind, bits, block, seed, STREAM_B2)
    q_b1 = q_b2 if reuse_b2 else quantize_grad(dH, PTQ, 8, 0, seed, STREAM_B1)
    return dict(q_x=q_x, q_w=q_w, q_b2=q_b2, q_b1=q_b1,
                grad_x=grad_x(q_b2, q_w), grad_w=grad_w(q_b1, q_x))
