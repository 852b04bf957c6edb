"""GPU parity: the CUDA library against the CPU oracle, through the C ABI.

Bars: bit-exact for integer work (PTQ / PSQ / deterministic codes, metadata,
sums, the integer contraction); BHQ codes agree on >= 99.99% of entries and
every mismatch is a +-1 flip at a stochastic-rounding boundary; gradients
agree within max |g - r| / max(|r|, 1e-3 ||r_row||_inf) <= 1e-3 with the
GPU's codes fed to the oracle's dequantize-then-multiply.
"""
import numpy as np
import pytest
import torch

import oracle as orc
from paper_2010_14298_gb300 import fqt
from paper_2010_14298_gb300 import workloads as wl
from gpu_util import (grad_rel_err, grouping_closed_form, oracle_groups_grad_x,
                      oracle_rows_grad_x, sr_boundary_distance,
                      to_dev)

pytestmark = [pytest.mark.gpu,
              pytest.mark.skipif(not torch.cuda.is_available(), reason="no GPU")]

GRAD_TOL = 1e-3


@pytest.fixture(scope="module", autouse=True)
def _lib():
    fqt.load()
    yield


# --------------------------------------------------------------------------
# Integer contraction core
# --------------------------------------------------------------------------
GEMM_CASES = [
    # M, N, K, a_kmajor, b_kmajor, a_bits, b_bits
    (300, 272, 208, 1, 0, 5, 8),      # grad_X layout, ragged tiles and K tail
    (64, 576, 5000, 0, 0, 8, 8),      # grad_W layout, split-K, exact chunks
    (128, 128, 64, 1, 1, 8, 8),
    (256, 160, 1040, 0, 1, 8, 4),
    (48, 32, 16, 1, 0, 2, 8),
    (1000, 64, 1024, 1, 0, 8, 8),
]


@pytest.mark.parametrize("M,N,K,ak,bk,ab,bb", GEMM_CASES)
def test_int_gemm_bit_exact(M, N, K, ak, bk, ab, bb):
    g = wl.rng(M * 7 + N * 3 + K)
    A = g.integers(0, 1 << ab, (M, K)).astype(np.uint8)
    B = g.integers(0, 1 << bb, (K, N)).astype(np.uint8)
    a_st = A if ak else np.ascontiguousarray(A.T)
    b_st = np.ascontiguousarray(B.T) if bk else B
    got = fqt.debug_int_gemm(torch.from_numpy(a_st).cuda(), ak, ab,
                             torch.from_numpy(b_st).cuda(), bk, bb, M, N, K)
    ref = orc.int_gemm(a_st, ak, b_st, bk, M, N, K, 1 << (ab - 1), 1 << (bb - 1))
    assert np.array_equal(got.cpu().numpy(), ref)


@pytest.mark.parametrize("K", [1024, 4096, 8192 + 64])
@pytest.mark.parametrize("fill", [(255, 255), (0, 0), (0, 255)])
def test_int_gemm_exact_at_extreme_magnitudes(K, fill):
    """Every product at its largest magnitude: partial sums reach the 2^24
    limit of exact fp32 accumulation inside each chunk."""
    M, N = 128, 128
    A = np.full((M, K), fill[0], dtype=np.uint8)
    B = np.full((K, N), fill[1], dtype=np.uint8)
    got = fqt.debug_int_gemm(torch.from_numpy(A).cuda(), 1, 8,
                             torch.from_numpy(B).cuda(), 0, 8, M, N, K)
    expect = K * (int(fill[0]) - 128) * (int(fill[1]) - 128)
    assert (got.cpu().numpy() == expect).all()


U8_GEMM_CASES = [
    # M, N, K, a_bits, b_bits: byte operands widened on chip (MN-major both)
    (64, 576, 5000, 8, 8),     # grad_W shape, split-K, exact chunks, K tail of 8 rows
    (128, 128, 64, 8, 8),
    (256, 160, 1040, 8, 4),    # ragged N tile, K tail of 16
    (48, 32, 16, 2, 8),        # one partial K block
    (96, 208, 3000, 5, 8),     # ragged M and N tiles
    (1024, 64, 777, 8, 8),
]


@pytest.mark.parametrize("M,N,K,ab,bb", U8_GEMM_CASES)
def test_int_gemm_u8_operands_bit_exact(M, N, K, ab, bb):
    """The split-K kernel reading byte codes and widening them on chip
    (grad_W's byte-operand path): bit-exact against the oracle's integer
    contraction, including K blocks past the end of the reduction (zero rows,
    where a zero byte would widen to -2^(b-1))."""
    g = wl.rng(M * 5 + N * 11 + K)
    A = g.integers(0, 1 << ab, (K, M)).astype(np.uint8)   # K x M (MN-major)
    B = g.integers(0, 1 << bb, (K, N)).astype(np.uint8)   # K x N (MN-major)
    got = fqt.debug_int_gemm_u8(torch.from_numpy(A).cuda(), ab, torch.from_numpy(B).cuda(), bb,
                                M, N, K)
    ref = orc.int_gemm(A, 0, B, 0, M, N, K, 1 << (ab - 1), 1 << (bb - 1))
    assert np.array_equal(got.cpu().numpy(), ref)


@pytest.mark.parametrize("K", [1024, 4096, 8192 + 64])
@pytest.mark.parametrize("fill", [(255, 255), (0, 0), (0, 255)])
def test_int_gemm_u8_exact_at_extreme_magnitudes(K, fill):
    M, N = 128, 128
    A = np.full((K, M), fill[0], dtype=np.uint8)
    B = np.full((K, N), fill[1], dtype=np.uint8)
    got = fqt.debug_int_gemm_u8(torch.from_numpy(A).cuda(), 8, torch.from_numpy(B).cuda(), 8,
                                M, N, K)
    expect = K * (int(fill[0]) - 128) * (int(fill[1]) - 128)
    assert (got.cpu().numpy() == expect).all()


@pytest.mark.parametrize("cfg", ["ffn-up", "conv"])
def test_grad_w_byte_operands_equal_carriers(cfg):
    """grad_W from byte-only code sets (Q_b1 and X~ without fp16 carriers)
    equals grad_W from the carriers bit for bit: the same exact integer
    partials, the same reduction."""
    g = wl.rng(808)
    if cfg == "ffn-up":
        n, c, d = 4096, 1024, 512
    else:
        n, c, d = 20000, 64, 576
    dH = wl.random_grad(g, n, c, sigma=1.0)
    X = g.uniform(-1, 1, (n, d)).astype(np.float32)
    dev = lambda a: to_dev(a, "f32")
    qx_c = fqt.quantize_act(dev(X), 8)
    q2, q1_c = fqt.quantize_grad(dev(dH), orc.BHQ, 5, 16, 17)
    qx_b = fqt.QTensor.empty(n, d, orc.PTQ, 8, 0, False, True, "cuda", u8=True, f16=False)
    fqt.quantize_act(dev(X), 8, out=qx_b)
    q1_b = fqt.QTensor.empty(n, c, orc.PTQ, 8, 0, False, True, "cuda", u8=True, f16=False)
    fqt.quantize_grad(dev(dH), orc.BHQ, 5, 16, 17, q_b2=q2, q_b1=q1_b)
    _, gw_c = fqt.linear_backward(q2, q1_c, qx_c, None, grad_x=False, grad_w=True)
    _, gw_b = fqt.linear_backward(q2, q1_b, qx_b, None, grad_x=False, grad_w=True)
    torch.cuda.synchronize()
    assert torch.equal(q1_b.codes, q1_c.codes) if q1_c.codes is not None else True
    assert torch.equal(gw_b, gw_c)


# --------------------------------------------------------------------------
# Quantizers
# --------------------------------------------------------------------------
def _check_b1(q1_gpu, dH, seed):
    r1 = orc.quantize_grad(dH, orc.PTQ, 8, 0, seed, orc.STREAM_B1)
    h1 = q1_gpu.to_numpy()
    assert np.array_equal(h1["codes"], r1["codes"])
    assert np.array_equal(h1["inv_s"], r1["inv_s"])
    assert np.array_equal(h1["zero"], r1["zero"])
    assert np.array_equal(h1["col_sum"], r1["codes"].astype(np.int64).sum(0))


# BHQ codes of every case compared in this module: the >= 99.99% agreement
# bar is a rate, so it is applied to each case of at least AGREE_MIN codes on
# its own and to the pool of all cases (test_bhq_code_agreement_pooled).
AGREE_MIN = 10_000
_BHQ_POOL = {"codes": 0, "flips": 0}


def _check_bhq_codes(got, ref, v, seed, stream=0):
    diff = got.astype(np.int64) - ref.astype(np.int64)
    flips = int((diff != 0).sum())
    _BHQ_POOL["codes"] += diff.size
    _BHQ_POOL["flips"] += flips
    # the transform rounds differently on the two sides (fp32 on the GPU,
    # double rounded to fp32 in the oracle): a mismatch is a +-1 flip where
    # v sits at its SR threshold
    assert np.abs(diff).max(initial=0) <= 1
    if diff.size >= AGREE_MIN:
        assert flips <= 1e-4 * diff.size, flips / diff.size
    idx = np.flatnonzero(diff.ravel())
    if idx.size:
        dist = sr_boundary_distance(v.ravel()[idx], seed, stream, idx)
        assert dist.max() <= 256, dist.max()  # within 2^-8 bin of the threshold


QUANT_CASES = [(0, None, orc.PTQ, 8, 0), (0, None, orc.PSQ, 8, 0),
               (0, None, orc.BHQ, 5, 16), (1, 2, orc.PTQ, 4, 0),
               (1, 2, orc.PSQ, 5, 0), (1, 2, orc.BHQ, 8, 16),
               (2, 1, orc.BHQ, 5, 8), (2, 1, orc.BHQ, 5, 64),
               (3, 64, orc.PSQ, 5, 0), (3, 64, orc.BHQ, 5, 16),
               (3, 64, orc.PTQ, 8, 0)]


@pytest.mark.parametrize("cfg,small,kind,bits,block", QUANT_CASES)
def test_quantize_grad_matches_oracle(cfg, small, kind, bits, block):
    kw = {}
    if cfg in (1, 2):
        kw["batch"] = small
    elif cfg == 3:
        kw["rows"] = small
    seed = 1234567
    for L in wl.config(cfg, **kw):
        dH = L.dH
        q2, q1 = fqt.quantize_grad(to_dev(dH, L.dtype), kind, bits, block, seed)
        ref = orc.quantize_grad(dH, kind, bits, block, seed, orc.STREAM_B2,
                                want_v=True)
        h2 = q2.to_numpy()
        assert np.array_equal(h2["row_sum"], h2["codes"].astype(np.int64).sum(1))
        if kind == orc.BHQ:
            assert np.array_equal(h2["lead"], ref["lead"])
            _check_bhq_codes(h2["codes"], ref["codes"], ref["v"], seed)
            assert np.allclose(h2["inv_s"], ref["inv_s"], rtol=1e-6, atol=0)
            assert np.allclose(h2["zero"], ref["zero"], rtol=1e-5, atol=1e-4)
        else:
            assert np.array_equal(h2["codes"], ref["codes"])
            assert np.array_equal(h2["inv_s"], ref["inv_s"])
            assert np.array_equal(h2["zero"], ref["zero"])
        _check_b1(q1, dH, seed)


@pytest.mark.parametrize("C,block,dtype", [(4096, 16, "f32"), (4096, 4, "f32"),
                                            (4096, 16, "bf16"), (2048, 8, "f32"),
                                            (512, 16, "bf16"), (1024, 4, "f32")])
def test_bhq_two_pass_widths_match_oracle(C, block, dtype):
    """The two-pass BHQ quantizer at the widths of its statistics pass: one
    warp per row group (C <= 128), a team of C / 256 warps (up to 2048), and
    a team of 8 warps over two column halves (C = 4096, the FFN's hidden
    width); ragged final block."""
    g = wl.rng(C + block)
    n = 37 * block + 3
    dH = wl.random_grad(g, n, C, sigma=1.3)
    if dtype == "bf16":
        dH = torch.from_numpy(dH).to(torch.bfloat16).float().numpy()
    seed = 4242
    q2, q1 = fqt.quantize_grad(to_dev(dH, dtype), orc.BHQ, 5, block, seed)
    ref = orc.quantize_grad(dH, orc.BHQ, 5, block, seed, orc.STREAM_B2, want_v=True)
    h2 = q2.to_numpy()
    assert np.array_equal(h2["lead"], ref["lead"])
    _check_bhq_codes(h2["codes"], ref["codes"], ref["v"], seed)
    assert np.allclose(h2["inv_s"], ref["inv_s"], rtol=1e-6, atol=0)
    assert np.allclose(h2["zero"], ref["zero"], rtol=1e-5, atol=1e-4)
    assert np.array_equal(h2["row_sum"], h2["codes"].astype(np.int64).sum(1))
    _check_b1(q1, dH, seed)


@pytest.mark.parametrize("kind,bits,block", [(orc.PTQ, 4, 0), (orc.PSQ, 8, 0),
                                             (orc.BHQ, 5, 16), (orc.BHQ, 5, 64)])
def test_fp16_carriers_encode_the_codes(kind, bits, block):
    """codes_f16 holds code - 2^(b-1) exactly, for both code sets."""
    L = wl.config(2, batch=1)[0]
    q2, q1 = fqt.quantize_grad(to_dev(L.dH), kind, bits, block, 9)
    for q, b in ((q2, bits), (q1, 8)):
        want = q.codes.to(torch.int32) - (1 << (b - 1))
        got = q.codes16.float()
        assert torch.equal(got, want.float())
    qx = fqt.quantize_act(to_dev(L.X), 8)
    assert torch.equal(qx.codes16.float(), qx.codes.float() - 128)


def test_quantize_fwd_matches_oracle():
    L = wl.config(1, batch=2)[0]
    for M in (L.X, L.W):
        q = fqt.quantize_act(to_dev(M), 8, row_sum=True)
        ref = orc.quantize_fwd(M, 8)
        h = q.to_numpy()
        assert np.array_equal(h["codes"], ref["codes"])
        assert np.array_equal(h["inv_s"], ref["inv_s"])
        assert np.array_equal(h["zero"], ref["zero"])
        assert np.array_equal(h["col_sum"], ref["codes"].astype(np.int64).sum(0))
        assert np.array_equal(h["row_sum"], ref["codes"].astype(np.int64).sum(1))


def test_quantize_fwd_bf16():
    L = wl.config(3, rows=64)[0]
    q = fqt.quantize_weight(to_dev(L.W, "bf16"), 8)
    ref = orc.quantize_fwd(L.W, 8)
    assert np.array_equal(q.codes.cpu().numpy(), ref["codes"])


# --------------------------------------------------------------------------
# The whole backward
# --------------------------------------------------------------------------
def _backward(L, kind, bits, block, seed=3, reuse=False):
    dev = lambda a: to_dev(a, L.dtype)
    qx = fqt.quantize_act(dev(L.X), 8)
    qw = fqt.quantize_weight(dev(L.W), 8)
    q2, q1 = fqt.quantize_grad(dev(L.dH), kind, bits, block, seed,
                               with_b1=not reuse, b2_col_sum=reuse)
    gx, gw = fqt.linear_backward(q2, q1, qx, qw)
    torch.cuda.synchronize()
    return qx, qw, q2, q1, gx.cpu().numpy(), gw.cpu().numpy()


BACKWARD_CASES = [(0, None, orc.PTQ, 8, 0), (0, None, orc.PSQ, 8, 0),
                  (0, None, orc.BHQ, 5, 16), (1, 2, orc.PTQ, 4, 0),
                  (1, 2, orc.BHQ, 5, 16), (2, 1, orc.BHQ, 5, 8),
                  (2, 1, orc.BHQ, 5, 32), (2, 1, orc.BHQ, 5, 64),
                  (2, 1, orc.BHQ, 4, 128), (0, None, orc.BHQ, 5, 2),
                  (3, 128, orc.BHQ, 5, 16), (3, 128, orc.BHQ, 8, 16),
                  (3, 128, orc.PTQ, 8, 0)]


@pytest.mark.parametrize("cfg,small,kind,bits,block", BACKWARD_CASES)
def test_linear_backward_matches_oracle(cfg, small, kind, bits, block):
    kw = {}
    if cfg in (1, 2):
        kw["batch"] = small
    elif cfg == 3:
        kw["rows"] = small
    for L in wl.config(cfg, **kw):
        qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, block)
        h2, h1, hx, hw = q2.to_numpy(), q1.to_numpy(), qx.to_numpy(), qw.to_numpy()
        ref_x = orc.grad_x(h2, hw)
        ref_w = orc.grad_w(h1, hx)
        assert grad_rel_err(gx, ref_x) <= GRAD_TOL
        assert grad_rel_err(gw, ref_w) <= GRAD_TOL


RESNET50 = wl.config(4, batch=1)


@pytest.mark.parametrize("idx", range(len(RESNET50)), ids=[L.name.split(":")[1] for L in RESNET50])
def test_resnet50_sweep_layer_matches_oracle(idx):
    """Every layer of the ResNet-50 sweep (batch 1; the stem's D and the fc's
    C zero-padded to multiples of 16): BHQ-5/16 codes against the oracle's,
    grad_X and grad_W against the oracle's dequantize-then-multiply of the
    GPU's codes."""
    L = RESNET50[idx]
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, 5, 16)
    h2 = q2.to_numpy()
    ref = orc.quantize_grad(L.dH, orc.BHQ, 5, 16, 3, orc.STREAM_B2, want_v=True)
    _check_bhq_codes(h2["codes"], ref["codes"], ref["v"], 3)
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL
    assert grad_rel_err(gw, orc.grad_w(q1.to_numpy(), qx.to_numpy())) <= GRAD_TOL


@pytest.mark.parametrize("N,block", [(256, 8), (200, 64), (131, 128), (77, 16)])
def test_bhq_offsets_match_oracle(N, block):
    """The reflected per-row terms of the grad_X epilogue against the
    oracle's reflection (Sec. 4.2) of the GPU's own zero points and row sums:
    2^(b-1) + z' = m + d with m the integer nearest its fp32 sum,
    hz = Q_blk d and hr = Q_blk (row_sum - C 2^(b-1) + C m)."""
    g = wl.rng(N + block)
    C, bits = 64, 5
    dH = wl.random_grad(g, N, C, outlier_frac=0.1)
    q2, _ = fqt.quantize_grad(to_dev(dH), orc.BHQ, bits, block, 9, with_b1=False)
    zero32 = q2.zero.cpu().numpy()
    rsum = q2.row_sum.cpu().numpy().astype(np.float64)
    lead = q2.lead.cpu().numpy()
    hz, hr = q2.hz.cpu().numpy(), q2.hr.cpu().numpy()
    oa = 2 ** (bits - 1)
    m = np.rint(np.float32(oa) + zero32).astype(np.float64)  # ties to even
    d = oa + zero32.astype(np.float64) - m
    R = rsum - C * oa + C * m
    assert np.all(np.abs(d) <= 0.5 + 1e-6)
    for b0 in range(0, N, block):
        nb = min(block, N - b0)
        Q = orc.householder(nb, int(lead[b0 // block])) if nb > 1 else np.eye(1)
        for got, x in ((hz, d[b0:b0 + nb]), (hr, R[b0:b0 + nb])):
            ref = Q @ x
            tol = 2.0 ** -23 * np.abs(ref) + 2.0 ** -36 * np.abs(x).max()
            assert np.all(np.abs(got[b0:b0 + nb] - ref) <= tol)


@pytest.mark.parametrize("cfg,small", [(0, None), (1, 2), (2, 1), (3, 128)])
def test_linear_forward_matches_oracle(cfg, small):
    """H = X~ W~^T (Sec. 2.1) through the same contraction core, against the
    oracle's dequantize-then-multiply of the GPU's forward codes."""
    kw = {}
    if cfg in (1, 2):
        kw["batch"] = small
    elif cfg == 3:
        kw["rows"] = small
    for L in wl.config(cfg, **kw):
        dev = lambda a: to_dev(a, L.dtype)
        qx = fqt.quantize_act(dev(L.X), 8, row_sum=True)
        qw = fqt.quantize_weight(dev(L.W), 8, row_sum=True)
        H = fqt.linear_forward(qx, qw)
        torch.cuda.synchronize()
        hx, hw = qx.to_numpy(), qw.to_numpy()
        assert np.array_equal(hx["row_sum"], hx["codes"].astype(np.int64).sum(axis=1))
        ref = orc.matmul(orc.dequant(hx), np.ascontiguousarray(orc.dequant(hw).T))
        assert H.shape == (L.N, L.W.shape[0])
        assert grad_rel_err(H.cpu().numpy(), ref) <= GRAD_TOL


def _offset_rows(g, n, c, rows, base=50.0, spread=1e-4):
    """Rows of one sign with a tiny range: their zero points put the row
    offset m far beyond the fp32 form of the contraction."""
    dH = wl.random_grad(g, n, c, sigma=1.0)
    for i, r in enumerate(rows):
        dH[r] = (base if i % 2 == 0 else -0.4 * base) + spread * g.standard_normal(c)
    return dH


@pytest.mark.parametrize("kind,bits,block", [(orc.BHQ, 5, 16), (orc.BHQ, 4, 2),
                                             (orc.BHQ, 5, 128), (orc.PSQ, 8, 0),
                                             (orc.PSQ, 4, 0)])
def test_tiles_outside_the_fp32_form(kind, bits, block):
    """Tiles with a row whose offset m exceeds the fp32 form are stored raw
    by the contraction and finished by the tile pass (int64 integer parts,
    float-float reflection); the other tiles stay in the fused epilogue."""
    g = wl.rng(330 + bits + block)
    n, c, d = 300, 64, 208  # row tiles 0..127, 128..255, 256..299; ragged columns
    dH = _offset_rows(g, n, c, [10, 140, 299], base=5000.0, spread=1e-2)
    X = g.uniform(-1, 1, (n, d)).astype(np.float32)
    W = (0.05 * g.standard_normal((c, d))).astype(np.float32)
    L = wl.Layer("offsets", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, block)
    h2, hw = q2.to_numpy(), qw.to_numpy()
    m = np.rint(np.float32(2 ** (bits - 1)) + h2["zero"].astype(np.float32))
    nb = max(block, 1)
    lim = 2.0 ** 24 / (2.0 + np.sqrt(nb)) if nb > 1 else 2.0 ** 24
    mmax = np.floor(lim / (c * 2.0 ** 7)) - 2 ** (bits - 1) - 1
    assert np.abs(m).max() > mmax  # at least one tile leaves the fp32 form
    assert grad_rel_err(gx, orc.grad_x(h2, hw)) <= GRAD_TOL


@pytest.mark.parametrize("kind,bits,block,c,raw", [(orc.PSQ, 8, 0, 2048, True),
                                                   (orc.PTQ, 8, 0, 3072, True),
                                                   (orc.BHQ, 8, 16, 2048, True),
                                                   (orc.BHQ, 5, 16, 2048, True),
                                                   (orc.BHQ, 5, 128, 1024, False)])
def test_tiles_outside_the_int32_form(kind, bits, block, c, raw):
    """Long reductions (two or three exact chunks with 8-bit codes; one chunk
    but no fp32 form with BHQ-5): the tile of a row whose offset m exceeds
    the int32 form keeps its products P as int32 bit patterns and the CTA's
    final pass finishes it in int64; a tile with a moderate offset stays in
    the int32 form; the rest are ordinary.  Blocks of 128 rows spread a
    row's offset over the block (every tile stays in the int32 form)."""
    g = wl.rng(440 + bits + block + c // 1024)
    n, d = 300, 208  # row tiles 0..127, 128..255, 256..299; ragged columns
    dH = wl.random_grad(g, n, c, sigma=1.0)
    if kind == orc.PTQ:
        dH = (3000.0 + 1e-2 * g.standard_normal((n, c))).astype(np.float32)
    else:
        dH[10] = 5000.0 + 1e-2 * g.standard_normal(c)        # far beyond the int32 form
        dH[140] = 6.0 + 0.5 * g.standard_normal(c)           # moderate offset
        dH[299] = -3000.0 + 1e-2 * g.standard_normal(c)      # ragged last tile
        dH = dH.astype(np.float32)
    X = g.uniform(-1, 1, (n, d)).astype(np.float32)
    W = (0.05 * g.standard_normal((c, d))).astype(np.float32)
    L = wl.Layer("offsets-long", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, block)
    h2, hw = q2.to_numpy(), qw.to_numpy()
    m = np.rint(np.float32(2 ** (bits - 1)) + h2["zero"].astype(np.float32))
    nb = max(block, 1)
    lim = (2.0 ** 31 - 1) / (2.0 + np.sqrt(nb)) if nb > 1 else 2.0 ** 31 - 1
    mmax32 = np.floor(lim / (c * 2.0 ** 7)) - 2 ** (bits - 1) - 1
    assert (np.abs(m).max() > mmax32) == raw  # whether a tile leaves the int32 form
    assert np.isfinite(gx).all()
    assert grad_rel_err(gx, orc.grad_x(h2, hw)) <= GRAD_TOL


def test_per_tensor_offset_sends_every_tile_to_the_tile_pass():
    """PTQ of an all-positive dH with a tiny range: one zero point for all
    rows, so every tile of grad_X -- and every tile of the forward for an X
    of that kind -- is finished by the tile pass."""
    g = wl.rng(341)
    n, c, d = 260, 64, 144
    dH = (50.0 + 1e-4 * g.standard_normal((n, c))).astype(np.float32)
    X = (20.0 + 1e-3 * g.standard_normal((n, d))).astype(np.float32)
    W = (0.05 * g.standard_normal((c, d))).astype(np.float32)
    L = wl.Layer("ptq-offset", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.PTQ, 5, 0)
    assert grad_rel_err(gx, orc.grad_x(q2.to_numpy(), qw.to_numpy())) <= GRAD_TOL
    qxr = fqt.quantize_act(to_dev(X), 8, row_sum=True)
    qwr = fqt.quantize_weight(to_dev(W), 8, row_sum=True)
    H = fqt.linear_forward(qxr, qwr)
    torch.cuda.synchronize()
    hx, hwr = qxr.to_numpy(), qwr.to_numpy()
    ref = orc.matmul(orc.dequant(hx), np.ascontiguousarray(orc.dequant(hwr).T))
    assert grad_rel_err(H.cpu().numpy(), ref) <= GRAD_TOL


def test_ptq_codes_reused_for_grad_w():
    L = wl.config(0)[0]
    qx, qw, q2, q1, gx, gw = _backward(L, orc.PTQ, 8, 0, reuse=True)
    assert q1 is None
    ref_w = orc.grad_w(q2.to_numpy(), qx.to_numpy())
    assert grad_rel_err(gw, ref_w) <= GRAD_TOL


@pytest.mark.parametrize("cfg,kind,bits,block", [(1, orc.BHQ, 5, 16),
                                                 (1, orc.PSQ, 4, 0),
                                                 (2, orc.BHQ, 5, 16)])
def test_full_size_sampled(cfg, kind, bits, block):
    """Full-size workloads in the bench's launch configuration: codes of all
    rows, grad_X on sampled row blocks, grad_W on sampled columns."""
    L = wl.config(cfg)[0]
    qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, block, seed=11)
    h2, h1, hx, hw = q2.to_numpy(), q1.to_numpy(), qx.to_numpy(), qw.to_numpy()
    ref2 = orc.quantize_grad(L.dH, kind, bits, block, 11, orc.STREAM_B2,
                             want_v=True)
    if kind == orc.BHQ:
        _check_bhq_codes(h2["codes"], ref2["codes"], ref2["v"], 11)
    else:
        assert np.array_equal(h2["codes"], ref2["codes"])
    _check_b1(q1, L.dH, 11)
    g = wl.rng(5)
    rows = np.sort(g.choice(L.N, 96, replace=False))
    ref_x = oracle_rows_grad_x(h2, hw, h2["codes"], rows)
    assert grad_rel_err(gx[rows], ref_x) <= GRAD_TOL
    cols = np.sort(g.choice(L.D, 32, replace=False))
    deq1 = orc.dequant(h1)
    deqx = orc.dequant(hx)[:, cols]
    ref_w = orc.matmul(deq1, deqx, a_trans=True)
    assert grad_rel_err(gw[:, cols], ref_w) <= GRAD_TOL


# --------------------------------------------------------------------------
# Edge cases and device-side status
# --------------------------------------------------------------------------
@pytest.mark.parametrize("N", [1, 5, 17, 33])
@pytest.mark.parametrize("kind,block", [(orc.PSQ, 0), (orc.BHQ, 16),
                                        (orc.BHQ, 64), (orc.PTQ, 0)])
def test_ragged_and_tiny(N, kind, block):
    g = wl.rng(N)
    dH = wl.random_grad(g, N, 48, outlier_frac=0.2)
    X = g.uniform(-1, 1, (N, 32)).astype(np.float32)
    W = g.standard_normal((48, 32)).astype(np.float32)
    L = wl.Layer("edge", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, kind, 5, block)
    ref = orc.quantize_grad(dH, kind, 5, block, 3, orc.STREAM_B2, want_v=True)
    if kind == orc.BHQ:
        _check_bhq_codes(q2.codes.cpu().numpy(), ref["codes"], ref["v"], 3)
    else:
        assert np.array_equal(q2.codes.cpu().numpy(), ref["codes"])
    h2, h1 = q2.to_numpy(), q1.to_numpy()
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL
    assert grad_rel_err(gw, orc.grad_w(h1, qx.to_numpy())) <= GRAD_TOL


@pytest.mark.parametrize("C,N,block,dtype", [(64, 200, 16, "f32"), (64, 77, 8, "bf16"),
                                             (128, 130, 16, "f32"), (256, 45, 8, "bf16"),
                                             (64, 1000, 32, "f32"), (256, 300, 4, "f32")])
def test_warp_quantizer_shapes(C, N, block, dtype):
    """Shapes of the warp-per-block BHQ quantizer (rows of 64/128/256 columns,
    ragged last block, bf16 input): codes against the oracle and the whole
    backward against the oracle's dequantize-then-multiply."""
    g = wl.rng(C + N + block)
    dH = wl.random_grad(g, N, C, outlier_frac=0.1)
    if dtype == "bf16":
        dH = wl.to_bf16_values(dH)
    X = g.uniform(-1, 1, (N, 48)).astype(np.float32)
    W = g.standard_normal((C, 48)).astype(np.float32)
    L = wl.Layer("warp", dH, X, W, dtype, [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, 5, block)
    ref = orc.quantize_grad(dH, orc.BHQ, 5, block, 3, orc.STREAM_B2, want_v=True)
    _check_bhq_codes(q2.codes.cpu().numpy(), ref["codes"], ref["v"], 3)
    assert np.array_equal(q2.lead.cpu().numpy(), ref["lead"])
    _check_b1(q1, dH, 3)
    h2, h1 = q2.to_numpy(), q1.to_numpy()
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL
    assert grad_rel_err(gw, orc.grad_w(h1, qx.to_numpy())) <= GRAD_TOL


@pytest.mark.parametrize("N,C,D", [(1000, 16, 48), (333, 48, 208), (4097, 64, 576),
                                   (64, 256, 256), (2051, 32, 1024)])
def test_grad_w_shapes(N, C, D):
    """grad_W through the one-CTA-per-K-range kernel at ragged K, C < 64 and
    several D tiles, against the oracle."""
    g = wl.rng(N + C + D)
    dH = wl.random_grad(g, N, C)
    X = g.uniform(-1, 1, (N, D)).astype(np.float32)
    W = g.standard_normal((C, D)).astype(np.float32)
    L = wl.Layer("gw", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.PSQ, 5, 0)
    assert grad_rel_err(gw, orc.grad_w(q1.to_numpy(), qx.to_numpy())) <= GRAD_TOL


def test_zero_and_constant_gradients():
    dH = np.zeros((64, 32), dtype=np.float32)
    dH[10] = 1.5
    dH[40:48] = -2.0
    for kind, block in ((orc.PTQ, 0), (orc.PSQ, 0), (orc.BHQ, 16)):
        q2, q1 = fqt.quantize_grad(to_dev(dH), kind, 4, block, 0)
        ref = orc.quantize_grad(dH, kind, 4, block, 0)
        assert np.array_equal(q2.codes.cpu().numpy(), ref["codes"])
        assert np.allclose(q2.inv_s.cpu().numpy(), ref["inv_s"], rtol=1e-6)


def test_empty_batch_is_a_no_op():
    dH = torch.zeros((0, 64), device="cuda")
    q2, q1 = fqt.quantize_grad(dH, orc.PSQ, 5, 0, 0)
    assert q2.codes.shape == (0, 64)


def test_nonfinite_input_is_reported_on_sync():
    dH = np.ones((32, 64), dtype=np.float32)
    dH[3, 5] = np.nan
    ws = fqt.Workspace(32, 64, 16)
    fqt.quantize_grad(to_dev(dH), orc.PSQ, 5, 0, 0, ws=ws)
    assert fqt.sync_status(ws) == 4
    assert fqt.sync_status(ws) == 0  # cleared
    dH[3, 5] = np.inf
    fqt.quantize_act(to_dev(dH), 8, ws=ws)
    assert fqt.sync_status(ws) == 4


def test_same_seed_same_codes_other_seed_other_codes():
    L = wl.config(0)[0]
    a, _ = fqt.quantize_grad(to_dev(L.dH), orc.BHQ, 5, 16, 77)
    b, _ = fqt.quantize_grad(to_dev(L.dH), orc.BHQ, 5, 16, 77)
    c, _ = fqt.quantize_grad(to_dev(L.dH), orc.BHQ, 5, 16, 78)
    assert torch.equal(a.codes, b.codes)
    assert not torch.equal(a.codes, c.codes)


def test_argument_errors():
    dH = torch.zeros((16, 12), device="cuda")  # C % 8 != 0
    with pytest.raises(fqt.FqtError) as e:
        fqt.quantize_grad(dH, orc.PSQ, 5, 0, 0)
    assert e.value.status == 2
    with pytest.raises(fqt.FqtError) as e:
        fqt.quantize_grad(torch.zeros((16, 16), device="cuda"), orc.BHQ, 5, 3, 0)
    assert e.value.status == 1


# --------------------------------------------------------------------------
# Adaptive BHQ groups (App. D.5; BHQ with block 0)
# --------------------------------------------------------------------------
def _adaptive_cases():
    g = wl.rng(300)
    out = []
    for n, c in ((1, 64), (2, 64), (7, 128), (130, 64), (4097, 64), (5000, 256)):
        out.append((f"random-{n}x{c}", wl.random_grad(g, n, c, sigma=2.0, outlier_frac=0.05)))
    eq = np.zeros((64, 64), np.float32)
    eq[:, 7] = 2.5
    eq[1::2, 7] = -2.5
    out.append(("equal-rows-64", eq))
    out.append(("cfg0-128", wl.config(0)[0].dH[:, :128].copy()))
    out.append(("cfg1-b2", wl.config(1, batch=2)[0].dH))
    out.append(("cfg2-b1", wl.config(2, batch=1)[0].dH))
    # row scales spread over orders of magnitude: groups of 33 .. 64 rows
    # (a warp's quantizer, a CTA's fix-up) and of 65 .. 591 rows (a CTA each)
    ln = g.standard_normal((20000, 64)) * np.exp(3.0 * g.standard_normal((20000, 1)))
    out.append(("lognormal-rows-20000x64", ln.astype(np.float32)))
    # a few outlier rows among many small ones: a handful of groups of 250+
    ol = 1e-3 * g.standard_normal((6000, 128))
    ol[:5] *= 1e4
    out.append(("outliers-6000x128", ol.astype(np.float32)))
    return out


ADAPTIVE = _adaptive_cases()


@pytest.mark.parametrize("idx", range(len(ADAPTIVE)), ids=[a[0] for a in ADAPTIVE])
def test_bhq_grouping_matches_oracle(idx):
    """perm, gstart, gsize and G of the GPU grouping equal the oracle's."""
    name, dH = ADAPTIVE[idx]
    q2, _ = fqt.quantize_grad(to_dev(dH), orc.BHQ, 5, 0, seed=3, with_b1=False)
    torch.cuda.synchronize()
    h2 = q2.to_numpy()
    ref = orc.bhq_grouping(dH)
    assert h2["G"] == ref["G"]
    assert np.array_equal(h2["perm"], ref["perm"])
    assert np.array_equal(h2["gstart"], ref["gstart"])
    assert np.array_equal(h2["gsize"], ref["gsize"])


@pytest.mark.parametrize("idx", range(len(ADAPTIVE)), ids=[a[0] for a in ADAPTIVE])
@pytest.mark.parametrize("bits", [4, 5, 8])
def test_bhq_adaptive_backward_matches_oracle(idx, bits):
    """Codes (stored order) and Q_b1 against the oracle; grad_X (scattered
    back to dH's row order) and grad_W against the oracle's
    dequantize-then-multiply of the GPU codes."""
    name, dH = ADAPTIVE[idx]
    n, c = dH.shape
    g = wl.rng(n + c + bits)
    X = g.uniform(-1, 1, (n, 48)).astype(np.float32)
    W = (0.05 * g.standard_normal((c, 48))).astype(np.float32)
    L = wl.Layer(name, dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, bits, 0)
    ref = orc.quantize_grad(dH, orc.BHQ, bits, 0, 3, orc.STREAM_B2, want_v=True)
    h2 = q2.to_numpy()
    assert np.array_equal(h2["perm"], ref["perm"])
    _check_bhq_codes(h2["codes"], ref["codes"], ref["v"], 3)
    _check_b1(q1, dH, 3)
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL
    assert grad_rel_err(gw, orc.grad_w(q1.to_numpy(), qx.to_numpy())) <= GRAD_TOL


def test_bhq_adaptive_bf16_and_wide_rows():
    g = wl.rng(310)
    dH = wl.to_bf16_values(wl.random_grad(g, 900, 128, sigma=2.5, outlier_frac=0.1))
    X = g.uniform(-1, 1, (900, 64)).astype(np.float32)
    W = (0.05 * g.standard_normal((128, 64))).astype(np.float32)
    L = wl.Layer("bf16", dH, X, W, "bf16", [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, 5, 0)
    ref = orc.quantize_grad(dH, orc.BHQ, 5, 0, 3, orc.STREAM_B2, want_v=True)
    h2 = q2.to_numpy()
    assert np.array_equal(h2["perm"], ref["perm"])
    _check_bhq_codes(h2["codes"], ref["codes"], ref["v"], 3)
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL


def test_bhq_adaptive_large_offsets_take_the_exact_path():
    """Rows of one sign with a tiny range have offsets m far beyond the fp32
    form: the contraction leaves them raw and the group pass finishes them
    in int64 / float-float."""
    g = wl.rng(320)
    dH = wl.random_grad(g, 300, 64, sigma=1.0)
    dH[10] = 50.0 + 1e-4 * g.standard_normal(64)   # all positive, R ~ 5e-4
    dH[11] = -20.0 + 1e-3 * g.standard_normal(64)
    X = g.uniform(-1, 1, (300, 32)).astype(np.float32)
    W = (0.05 * g.standard_normal((64, 32))).astype(np.float32)
    L = wl.Layer("offsets", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, 5, 0)
    h2 = q2.to_numpy()
    m = np.rint(np.float32(16) + h2["zero"])
    # the fp32 form holds |m| <= 2^24 / (C 2^(bw-1)) - 2^(b-1) - 1 = 2031 here
    assert np.abs(m).max() > 2031
    assert grad_rel_err(gx, orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL


def test_bhq_adaptive_full_size_sampled():
    """The ResNet-18 conv workload at full size (131072 x 64): the grouping
    against its definition (closed form of the estimate, leads, cumulative
    rounding), grad_X on sampled whole groups."""
    L = wl.config(1)[0]
    qx, qw, q2, q1, gx, gw = _backward(L, orc.BHQ, 5, 0, seed=11)
    h2, hw = q2.to_numpy(), qw.to_numpy()
    n = L.N
    order, Ms, V, sizes = grouping_closed_form(L.dH)
    G = h2["G"]
    best = V.min()
    assert V[G - 1] <= best * (1 + 1e-12)
    if V[G - 1] > best:  # a near tie: the other choice is as good
        assert np.argmin(V) + 1 != G
    gs = h2["gstart"]
    assert np.all(gs[G:] == n) and np.all(np.diff(gs[:G + 1]) >= 1)
    assert np.array_equal(h2["perm"][gs[:G]], order[:G])
    e = sizes(G)
    assert np.array_equal(np.diff(gs[:G + 1]) - 1, np.diff(e))
    assert np.array_equal(np.sort(h2["perm"]), np.arange(n))
    g = wl.rng(7)
    big = np.argsort(-(np.diff(gs[:G + 1])))[:8]
    groups = np.unique(np.concatenate([big, g.choice(G, 56, replace=False)]))
    ref = oracle_groups_grad_x(h2, hw, groups)
    rows = np.array(sorted(ref))
    assert grad_rel_err(gx[rows], np.stack([ref[r] for r in rows])) <= GRAD_TOL


# --------------------------------------------------------------------------
# Per-sample power-of-two shift quantizer (Sec. 4.3; kind SHIFT)
# --------------------------------------------------------------------------
SHIFT_C = (64, 128, 256, 512, 1024)


def _shift_layers(cfg, small):
    kw = {}
    if cfg in (1, 2):
        kw["batch"] = small
    elif cfg in (0, 3):
        kw["rows"] = small
    return [L for L in wl.config(cfg, **kw) if L.C in SHIFT_C]


@pytest.mark.parametrize("cfg,small", [(0, None), (1, 2), (2, 1), (3, 256)])
@pytest.mark.parametrize("bits", [4, 5, 8])
def test_shift_quantizer_matches_oracle(cfg, small, bits):
    """Codes, shifts, scales and zero points bit for bit (both sides decide
    in fp32 with the same operations); the shifted grad_W operand and its
    column sums exactly."""
    for L in _shift_layers(cfg, small):
        q2, _ = fqt.quantize_grad(to_dev(L.dH, L.dtype), fqt.SHIFT, bits, 0, seed=5,
                                  with_b1=False)
        torch.cuda.synchronize()
        h2 = q2.to_numpy()
        ref = orc.quantize_grad(L.dH, orc.SHIFT, bits, 0, 5, orc.STREAM_B2)
        for key in ("codes", "inv_s", "zero", "shift"):
            assert np.array_equal(h2[key], ref[key]), key
        a = orc.shifted_codes(ref)
        assert np.array_equal(q2.shift16.float().cpu().numpy().astype(np.int64), a)
        assert np.array_equal(q2.shift_col_sum.cpu().numpy(), a.sum(axis=0))
        assert np.array_equal(h2["row_sum"], ref["codes"].astype(np.int64).sum(1))
        sc = q2.shift_scale.cpu().numpy()
        assert sc[1] == 0.0
        assert sc[0] == np.float32(ref["inv_s"][0] * np.float32(2.0 ** (int(ref["shift"][0]) - 4)))


@pytest.mark.parametrize("cfg,small", [(0, None), (1, 2), (2, 1), (3, 256)])
@pytest.mark.parametrize("bits", [4, 5, 8])
def test_shift_backward_matches_oracle(cfg, small, bits):
    """No bifurcation: the shift codes feed grad_X (as a per-row encoding)
    and grad_W (shifted integer accumulators, Sec. 4.3)."""
    for L in _shift_layers(cfg, small):
        dev = lambda x: to_dev(x, L.dtype)
        ws = fqt.Workspace(L.N, L.C, L.D)
        qx = fqt.quantize_act(dev(L.X), 8)
        qw = fqt.quantize_weight(dev(L.W), 8)
        q2, q1 = fqt.quantize_grad(dev(L.dH), fqt.SHIFT, bits, 0, seed=3, with_b1=False,
                                   ws=ws)
        gx, gw = fqt.linear_backward(q2, None, qx, qw, ws=ws)
        assert fqt.sync_status(ws) == 0
        h2, hx, hw = q2.to_numpy(), qx.to_numpy(), qw.to_numpy()
        assert grad_rel_err(gx.cpu().numpy(), orc.grad_x(h2, hw)) <= GRAD_TOL
        ref_w = orc.grad_w_shifted(h2, hx)
        assert grad_rel_err(gw.cpu().numpy(), ref_w) <= GRAD_TOL
        assert np.abs(ref_w - orc.grad_w(h2, hx)).max() <= 1e-9 * np.abs(ref_w).max()


@pytest.mark.parametrize("N,C", [(1, 64), (7, 128), (333, 256), (1000, 512), (65, 1024)])
def test_shift_shapes_ragged_and_bf16(N, C):
    g = wl.rng(N + C)
    dH = wl.to_bf16_values(wl.random_grad(g, N, C, sigma=2.5, outlier_frac=0.1))
    X = g.uniform(-1, 1, (N, 32)).astype(np.float32)
    W = (0.05 * g.standard_normal((C, 32))).astype(np.float32)
    qx = fqt.quantize_act(to_dev(X), 8)
    qw = fqt.quantize_weight(to_dev(W), 8)
    q2, _ = fqt.quantize_grad(to_dev(dH, "bf16"), fqt.SHIFT, 5, 0, seed=9, with_b1=False)
    gx, gw = fqt.linear_backward(q2, None, qx, qw)
    torch.cuda.synchronize()
    h2 = q2.to_numpy()
    ref = orc.quantize_grad(dH, orc.SHIFT, 5, 0, 9, orc.STREAM_B2)
    assert np.array_equal(h2["codes"], ref["codes"]) and np.array_equal(h2["shift"], ref["shift"])
    assert grad_rel_err(gx.cpu().numpy(), orc.grad_x(h2, qw.to_numpy())) <= GRAD_TOL
    assert grad_rel_err(gw.cpu().numpy(), orc.grad_w_shifted(h2, qx.to_numpy())) <= GRAD_TOL


def test_shift_with_a_bifurcated_q_b1_too():
    """The shift kind may still emit the 8-bit PTQ Q_b1 in the same pass."""
    L = wl.config(1, batch=2)[0]
    q2, q1 = fqt.quantize_grad(to_dev(L.dH), fqt.SHIFT, 5, 0, seed=3, with_b1=True)
    torch.cuda.synchronize()
    _check_b1(q1, L.dH, 3)


# --------------------------------------------------------------------------
# Implicit im2col operand (NEXT n3, the X~ side): NHWC codes, shifted loads
# --------------------------------------------------------------------------
def _conv_codes_as_im2col(q, x_shape, kh, kw, pad):
    """The im2col matrix of the GPU's NHWC codes (padding = code of 0.0)."""
    n, h, w, c = x_shape
    zc = int(q.col_sum[-1].item())  # the code of 0.0: the padding's code
    nhwc = (q.codes16.float().cpu().numpy().astype(np.int64)
            + (1 << (q.bits - 1))).reshape(n, h, w, c)
    full = np.full((n, h + 2 * pad, w + 2 * pad, c), zc, dtype=np.int64)
    full[:, pad:pad + h, pad:pad + w] = nhwc
    oh, ow = h + 2 * pad - kh + 1, w + 2 * pad - kw + 1
    cols = np.empty((n, oh, ow, kh, kw, c), dtype=np.int64)
    for i in range(kh):
        for j in range(kw):
            cols[:, :, :, i, j, :] = full[:, i:i + oh, j:j + ow, :]
    return cols.reshape(n * oh * ow, kh * kw * c), zc


@pytest.mark.parametrize("n,h,w,c,k,pad,dtype", [
    (2, 32, 32, 64, 3, 1, "f32"), (1, 32, 32, 128, 3, 1, "bf16"), (3, 8, 12, 16, 3, 1, "f32"),
    (2, 9, 9, 64, 3, 0, "f32"), (3, 7, 7, 512, 3, 1, "f32"), (2, 11, 10, 64, 5, 2, "f32"),
    (2, 6, 7, 64, 3, 2, "f32"), (2, 5, 5, 32, 1, 0, "f32"), (1, 9, 9, 512, 3, 0, "f32")])
def test_conv_quantizer_equals_the_im2col_quantizer(n, h, w, c, k, pad, dtype):
    """Codes, scale and im2col column sums of the implicit Q_f against the
    oracle's quantizer on the explicit im2col matrix; the kernel sizes and
    paddings span the column sums' border classes (pad < k - 1, = k - 1,
    > k - 1) and the per-tap fallback (9 x 9 classes of 512 channels)."""
    g = wl.rng(n * h + c + pad + 7 * k)
    x = g.uniform(-1, 1, (n, h, w, c)).astype(np.float32)
    x[0, 0, 0, :4] = 3.0  # the range is not symmetric
    if dtype == "bf16":
        x = wl.to_bf16_values(x)
    xi = wl.im2col_nhwc(x, k, k, 1, pad)
    ref = orc.quantize_fwd(xi, 8)
    q = fqt.quantize_act_conv(to_dev(x, dtype), k, k, pad, 8)
    torch.cuda.synchronize()
    assert q.shape == xi.shape
    got, zc = _conv_codes_as_im2col(q, x.shape, k, k, pad)
    assert np.array_equal(got, ref["codes"].astype(np.int64))
    assert np.array_equal(q.inv_s.cpu().numpy(), ref["inv_s"])
    assert np.array_equal(q.zero.cpu().numpy(), ref["zero"])
    assert np.array_equal(q.col_sum[:-1].cpu().numpy(), ref["codes"].astype(np.int64).sum(0))


@pytest.mark.parametrize("batch", [2, 128])
def test_conv_grad_w_equals_the_explicit_path(batch):
    """grad_W with X~ read as shifted NHWC boxes equals grad_W over the
    materialized im2col codes bit for bit (the contraction is exact), and the
    oracle within the tolerance (sampled columns at batch 128)."""
    g = wl.rng(400 + batch)
    x = g.uniform(-1, 1, (batch, 32, 32, 64)).astype(np.float32)
    xi = wl.im2col_nhwc(x, 3, 3, 1, 1)
    N = xi.shape[0]
    dH = g.standard_normal((N, 64)).astype(np.float32)
    dH[g.random(N) < 0.01] *= 100.0
    W = (np.sqrt(2.0 / 576) * g.standard_normal((64, 576))).astype(np.float32)
    qw = fqt.quantize_weight(to_dev(W), 8)
    q2, q1 = fqt.quantize_grad(to_dev(dH), orc.BHQ, 5, 16, seed=3)
    ws = fqt.Workspace(N, 64, 576)
    qx = fqt.quantize_act(to_dev(xi), 8)
    qc = fqt.quantize_act_conv(to_dev(x), 3, 3, 1, 8)
    _, gw = fqt.linear_backward(q2, q1, qx, qw, grad_x=False, ws=ws)
    _, gwc = fqt.linear_backward(q2, q1, qc, qw, grad_x=False, ws=ws)
    assert fqt.sync_status(ws) == 0
    gw, gwc = gw.cpu().numpy(), gwc.cpu().numpy()
    assert np.array_equal(gw, gwc)
    h1, hx = q1.to_numpy(), qx.to_numpy()
    cols = np.arange(576) if batch == 2 else np.sort(wl.rng(5).choice(576, 48, replace=False))
    ref = orc.matmul(orc.dequant(h1), orc.dequant(hx)[:, cols], a_trans=True)
    assert grad_rel_err(gwc[:, cols], ref) <= GRAD_TOL


@pytest.mark.parametrize("n,h,w,cin,cout,k,pad", [
    (2, 56, 56, 64, 64, 3, 1), (3, 28, 28, 128, 128, 3, 1), (4, 14, 14, 64, 256, 3, 1),
    (5, 7, 7, 128, 64, 3, 1), (2, 9, 11, 64, 128, 3, 1), (1, 64, 64, 64, 64, 3, 1),
    (2, 12, 96, 64, 64, 3, 1), (2, 14, 13, 64, 64, 5, 2), (2, 10, 10, 64, 512, 3, 2),
    (3, 9, 9, 64, 128, 1, 0), (2, 7, 7, 512, 512, 3, 1)])
def test_conv_grad_w_rows_in_blocks_equal_the_explicit_path(n, h, w, cin, cout, k, pad):
    """The implicit im2col X~ in the split-K tile kernel at the output-row
    widths of ResNet-50's 3 x 3 layers (56, 28, 14, 7) and ragged ones: K
    blocks of whole output rows padded to a power of two (64 / 32 / 16 / 8
    slots, rows past oh and slots past ow zero), bit for bit the explicit
    im2col grad_W; ow = 96 takes the one-range-per-CTA kernel.  5 x 5 / pad 2,
    pad 2 on 3 x 3 and 1 x 1 / pad 0 vary the padding correction's classes."""
    g = wl.rng(n * h * w + cin + cout + 11 * k + pad)
    x = g.uniform(-1, 1, (n, h, w, cin)).astype(np.float32)
    xi = wl.im2col_nhwc(x, k, k, 1, pad)
    N, D = xi.shape
    dH = g.standard_normal((N, cout)).astype(np.float32)
    dH[g.random(N) < 0.02] *= 50.0
    q2, q1 = fqt.quantize_grad(to_dev(dH), orc.BHQ, 5, 16, seed=9)
    ws = fqt.Workspace(N, cout, D)
    qx = fqt.quantize_act(to_dev(xi), 8)
    qc = fqt.quantize_act_conv(to_dev(x), k, k, pad, 8)
    _, gw = fqt.linear_backward(q2, q1, qx, None, grad_x=False, ws=ws)
    _, gwc = fqt.linear_backward(q2, q1, qc, None, grad_x=False, ws=ws)
    assert fqt.sync_status(ws) == 0
    assert torch.equal(gw, gwc)


# --------------------------------------------------------------------------
# Unbiasedness of the GPU quantizers over seeds (Sec. 3.3, 4.1-4.3; the
# premise of Thm 1): the mean of the dequantized GPU codes is dH, with the
# spread the exact per-code variances predict.
# --------------------------------------------------------------------------
def _code_moments(v, B):
    var = np.zeros(v.shape)
    for idx in np.ndindex(v.shape):
        var[idx] = orc.sr_moments(float(v[idx]), B)[1]
    return var


@pytest.mark.parametrize("kind,bits,block", [(orc.PSQ, 4, 0), (orc.BHQ, 4, 8), (orc.SHIFT, 4, 0)])
def test_gpu_quantizers_are_unbiased_monte_carlo(kind, bits, block):
    g = wl.rng(500 + kind)
    h = wl.random_grad(g, 16, 64, sigma=1.5, outlier_frac=0.1)
    B = (1 << bits) - 1
    ref = orc.quantize_grad(h, kind, bits, block, 0, want_v=True)
    vc = _code_moments(ref["v"], B)
    inv = ref["inv_s"].astype(np.float64)
    if kind == orc.BHQ:
        vd = np.zeros(h.shape)
        for b, r0 in enumerate(range(0, 16, block)):
            Q = orc.householder(block, int(ref["lead"][b]))
            vd[r0:r0 + block] = ((inv[r0:r0 + block, None] * Q) ** 2) @ vc[r0:r0 + block]
    else:
        vd = vc * (inv ** 2)[:, None]
    K = 512
    dH = to_dev(h)
    s1 = np.zeros(h.shape)
    s2 = np.zeros(h.shape)
    for seed in range(K):
        q2, _ = fqt.quantize_grad(dH, kind, bits, block, seed=seed + 77, with_b1=False)
        d = orc.dequant(q2.to_numpy())
        s1 += d
        s2 += d * d
    mean = s1 / K
    # the z bound needs the normal approximation of each entry's count of
    # round-ups: p (1 - p) K >= 8 (BHQ entries mix a block's codes: its
    # smallest code variance decides)
    if kind == orc.BHQ:
        vmin = np.zeros(h.shape)
        for r0 in range(0, 16, block):
            vmin[r0:r0 + block] = vc[r0:r0 + block].min(axis=0)
    else:
        vmin = vc
    live = (vd > 0) & (vmin * K >= 8)
    assert live.mean() > 0.5
    z = (mean - h)[live] / np.sqrt(vd[live] / K)
    assert np.abs(z).max() < 5.5
    emp = (s2 / K - mean ** 2).sum()
    assert emp / vd.sum() == pytest.approx(1.0, rel=0.12)


# --------------------------------------------------------------------------
# Full-size workloads of the transformer FFN pair and the ResNet-50 sweep,
# at the sizes the bench times (sampled outputs)
# --------------------------------------------------------------------------
def _grad_w_columns(h1: dict, hx: dict, cols: np.ndarray) -> np.ndarray:
    """The oracle's dequantize-then-multiply grad_W on a subset of the
    columns of a per-tensor X~ (its dequantization is column-separable); the
    double product of the two dequantized matrices is a BLAS dgemm here (the
    oracle's plain loop takes minutes at millions of rows)."""
    sub = dict(hx)
    sub["codes"] = np.ascontiguousarray(hx["codes"][:, cols])
    return orc.dequant(h1).T @ orc.dequant(sub)


def _sampled_check(L, kind, bits, block, seed, n_rows=96, n_cols=32):
    """Every code of Q_b2 and Q_b1 against the oracle's, grad_X on sampled
    rows (whole quantizer blocks) and grad_W on sampled columns against the
    oracle's dequantize-then-multiply of the GPU's codes."""
    qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, block, seed=seed)
    h2, h1, hx, hw = q2.to_numpy(), q1.to_numpy(), qx.to_numpy(), qw.to_numpy()
    ref2 = orc.quantize_grad(L.dH, kind, bits, block, seed, orc.STREAM_B2,
                             want_v=kind == orc.BHQ)
    if kind == orc.BHQ:
        _check_bhq_codes(h2["codes"], ref2["codes"], ref2["v"], seed)
        assert np.array_equal(h2["lead"], ref2["lead"])
    else:
        assert np.array_equal(h2["codes"], ref2["codes"])
        assert np.array_equal(h2["inv_s"], ref2["inv_s"])
        assert np.array_equal(h2["zero"], ref2["zero"])
    del ref2
    _check_b1(q1, L.dH, seed)
    ref_f = orc.quantize_fwd(L.X, 8)
    assert np.array_equal(hx["codes"], ref_f["codes"])
    del ref_f
    g = wl.rng(L.N + L.C + L.D)
    rows = np.sort(g.choice(L.N, min(n_rows, L.N), replace=False))
    rows = np.union1d(rows, [0, L.N - 1])  # the first and the ragged last block
    ref_x = oracle_rows_grad_x(h2, hw, h2["codes"], rows)
    assert grad_rel_err(gx[rows], ref_x) <= GRAD_TOL
    cols = np.sort(g.choice(L.D, min(n_cols, L.D), replace=False))
    cols = np.union1d(cols, [0, L.D - 1])
    assert grad_rel_err(gw[:, cols], _grad_w_columns(h1, hx, cols)) <= GRAD_TOL


_FFN = {}


def _ffn_layer(i):
    if not _FFN:
        _FFN.update(enumerate(wl.config(3)))
    return _FFN[i]


@pytest.mark.parametrize("kind,bits,block", [(orc.PTQ, 8, 0), (orc.PSQ, 5, 0),
                                             (orc.BHQ, 5, 16)])
@pytest.mark.parametrize("layer", [0, 1], ids=["ffn-up", "ffn-down"])
def test_ffn_full_size_sampled(layer, kind, bits, block):
    """The transformer FFN pair at 8192 tokens from bf16 tensors (C = 4096
    and 1024): the int64 and mixed epilogue forms, several exact chunks per
    split-K range of grad_W, at the shapes the bench times."""
    _sampled_check(_ffn_layer(layer), kind, bits, block, seed=13)


R50_FULL = ["conv1", "layer1.0.conv2", "layer1.0.conv3", "fc"]


@pytest.mark.parametrize("name", R50_FULL)
def test_resnet50_full_batch_layer_sampled(name):
    """Layers of the ResNet-50 sweep at batch 256: the stem (N = 3,211,264
    im2col rows, D 147 -> 160), a 3 x 3 and a 1 x 1 layer of stage 1
    (N = 802,816, C = 64 and 256) and the fc (C 1000 -> 1008); BHQ-5/16 with
    Q_b1, as the bench runs them."""
    shapes = wl.resnet50_shapes()
    i = [s.name for s in shapes].index(name)
    L = wl.resnet50_layer(shapes[i], 256, 1234 + 4 + i)
    _sampled_check(L, orc.BHQ, 5, 16, seed=3)


@pytest.mark.parametrize("kind,bits", [(orc.PTQ, 8), (orc.PSQ, 8), (orc.BHQ, 8)])
def test_grad_x_several_chunks_and_tiles_per_cta(kind, bits):
    """grad_X with two exact chunks per tile (8-bit codes, C = 2048) and at
    least three tiles per CTA (480 tiles): the accumulators are reused by
    later tiles while earlier tiles' chunks drain."""
    g = wl.rng(2048)
    n, c, d = 7680, 2048, 1024
    dH = wl.random_grad(g, n, c, sigma=1.5)
    X = g.standard_normal((n, d)).astype(np.float32)
    W = (0.02 * g.standard_normal((c, d))).astype(np.float32)
    L = wl.Layer("chunks", dH, X, W, "f32", [])
    qx, qw, q2, q1, gx, gw = _backward(L, kind, bits, 16 if kind == orc.BHQ else 0, seed=4)
    h2, hw = q2.to_numpy(), qw.to_numpy()
    rows = np.sort(wl.rng(7).choice(n, 160, replace=False))
    ref_x = oracle_rows_grad_x(h2, hw, h2["codes"], rows)
    assert grad_rel_err(gx[rows], ref_x) <= GRAD_TOL


# --------------------------------------------------------------------------
# Per-image samples (Sec. 4.1: a sample is one input's gradient)
# --------------------------------------------------------------------------
SAMPLE_CASES = [  # rows N, C, rows per sample, bits, dtype
    (2048, 64, 1024, 5, "f32"), (2048, 64, 1024, 8, "f32"), (3136 * 2, 256, 3136, 5, "f32"),
    (196 * 4, 1024, 196, 5, "bf16"), (49 * 3, 2048, 49, 4, "f32"), (600, 128, 1, 5, "f32"),
    (512, 512, 128, 8, "bf16"), (64 * 3, 4096, 64, 5, "bf16")]


@pytest.mark.parametrize("N,C,R,bits,dtype", SAMPLE_CASES)
def test_per_sample_psq_matches_oracle(N, C, R, bits, dtype):
    g = wl.rng(N + C + R)
    dH = wl.random_grad(g, N, C, sigma=1.5, outlier_frac=0.05)
    if dtype == "bf16":
        dH = wl.to_bf16_values(dH)
    q2, q1 = fqt.quantize_grad_samples(to_dev(dH, dtype), R, orc.PSQ, bits, seed=21)
    torch.cuda.synchronize()
    ref = orc.quantize_grad_samples(dH, R, orc.PSQ, bits, 0, seed=21)
    h2 = q2.to_numpy()
    assert np.array_equal(h2["codes"], ref["codes"])
    assert np.array_equal(h2["inv_s"], ref["inv_s_rows"])
    assert np.array_equal(h2["zero"], ref["zero_rows"])
    assert np.array_equal(h2["row_sum"], h2["codes"].astype(np.int64).sum(1))
    _check_b1(q1, dH, 21)
    assert q2.c_struct().rows_per_sample == R


def test_one_row_samples_equal_the_row_quantizer_on_the_gpu():
    """rows_per_sample = 1 (the per-sample code pass) against quantize_grad's
    PSQ (the staged row kernel): the same codes and metadata bit for bit."""
    L = wl.config(1, batch=1)[0]
    a2, a1 = fqt.quantize_grad_samples(to_dev(L.dH), 1, orc.PSQ, 5, seed=8)
    b2, b1 = fqt.quantize_grad(to_dev(L.dH), orc.PSQ, 5, 0, 8)
    for x, y in ((a2, b2), (a1, b1)):
        hx, hy = x.to_numpy(), y.to_numpy()
        for k in ("codes", "inv_s", "zero", "col_sum"):
            if hx.get(k) is not None and hy.get(k) is not None:
                assert np.array_equal(hx[k], hy[k]), k


def test_per_sample_backward_matches_oracle():
    """grad_X and grad_W of the ResNet-18 conv layer at batch 2 with per-image
    PSQ-5 (1024 rows per image): the PSQ epilogue reads the repeated
    per-row scalars."""
    L = wl.config(1, batch=2)[0]
    qx = fqt.quantize_act(to_dev(L.X), 8)
    qw = fqt.quantize_weight(to_dev(L.W), 8)
    q2, q1 = fqt.quantize_grad_samples(to_dev(L.dH), 1024, orc.PSQ, 5, seed=4)
    gx, gw = fqt.linear_backward(q2, q1, qx, qw)
    torch.cuda.synchronize()
    ref = orc.quantize_grad_samples(L.dH, 1024, orc.PSQ, 5, 0, seed=4)
    ref["codes"] = q2.to_numpy()["codes"]
    rx = orc.matmul(orc.dequant_samples(ref), orc.dequant(qw.to_numpy()))
    assert grad_rel_err(gx.cpu().numpy(), rx) <= GRAD_TOL
    assert grad_rel_err(gw.cpu().numpy(), orc.grad_w(q1.to_numpy(), qx.to_numpy())) <= GRAD_TOL


def test_per_sample_refusals():
    dH = torch.zeros((100, 64), device="cuda")
    with pytest.raises(fqt.FqtError) as e:
        fqt.quantize_grad_samples(dH, 30, orc.PSQ, 5)  # 100 rows are not whole samples
    assert e.value.status == 1
    with pytest.raises(fqt.FqtError) as e:
        fqt.quantize_grad_samples(dH, 10, orc.BHQ, 5)
    assert e.value.status == 2


def test_bhq_code_agreement_pooled():
    """The >= 99.99% BHQ code agreement over every case this module compared
    (cases below AGREE_MIN codes cannot show a 1e-4 rate on their own)."""
    if _BHQ_POOL["codes"] == 0:
        pytest.skip("no BHQ case ran")
    assert _BHQ_POOL["flips"] <= 1e-4 * _BHQ_POOL["codes"], _BHQ_POOL
