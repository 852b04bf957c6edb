"""Pins of the CPU oracle to what the paper and the mathematics fix.

None of these tests calls the CUDA library.  Each one checks the oracle
against something other than itself: published known answers, exact
expectations by enumeration of every rounding outcome, the paper's variance
expressions and bounds, the Householder identities, and special cases that
reduce to another quantizer or to a library routine.
"""
import os

import numpy as np
import pytest

import oracle as orc
from paper_2010_14298_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _moments(v: np.ndarray, B: int):
    """Exact mean and variance of every code, by enumerating all uniforms."""
    m = np.zeros(v.shape)
    var = np.zeros(v.shape)
    for idx in np.ndindex(v.shape):
        m[idx], var[idx] = orc.sr_moments(float(v[idx]), B)
    return m, var


def _blocks(n, nb):
    return [(r0, min(nb, n - r0)) for r0 in range(0, n, nb)]


# --------------------------------------------------------------------------
# Philox4x32-10 and the uniforms
# --------------------------------------------------------------------------
def test_philox_known_answers():
    rows = [l.split() for l in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt"))
            if l.strip() and not l.startswith("#")]
    assert len(rows) == 3
    for r in rows:
        vals = [int(x, 16) for x in r]
        assert orc.philox4x32_10(vals[:4], vals[4:6]) == tuple(vals[6:10])


def test_uniform_layout_reads_the_philox_block():
    seed, stream = 0x1234_5678_9ABC_DEF0, 1
    for q in (0, 1, 77, 1 << 33):
        w = orc.philox4x32_10([q & 0xFFFFFFFF, q >> 32, stream, 0],
                              [seed & 0xFFFFFFFF, seed >> 32])
        for i in range(8):
            expect = (w[i // 2] >> (16 * (i % 2))) & 0xFFFF
            assert orc.u16(seed, stream, 8 * q + i) == expect


def test_uniforms_are_uniform_and_streams_distinct():
    n = 1 << 16
    a = np.array([orc.u16(7, 0, i) for i in range(n)])
    b = np.array([orc.u16(7, 1, i) for i in range(n)])
    for u in (a, b):
        hist = np.bincount(u >> 10, minlength=64)
        chi2 = ((hist - n / 64) ** 2 / (n / 64)).sum()
        assert chi2 < 130  # df = 63; p(chi2 > 130) ~ 1e-6
    assert abs(np.corrcoef(a, b)[0, 1]) < 0.02
    assert (a != b).mean() > 0.99


# --------------------------------------------------------------------------
# Stochastic rounding (Sec. 3.3, App. D: E[SR(X)] = X, Var = p (1 - p))
# --------------------------------------------------------------------------
@pytest.mark.parametrize("v", [0.0, 0.25, 0.5, 1.0, 3.7, 12.999, 100.3125,
                               254.5, 254.99, 255.0, 1e-7, 17.000001])
def test_sr_moments_match_the_definition(v):
    B = 255
    m, var = orc.sr_moments(v, B)
    v32 = float(np.float32(v))
    assert v32 - 2.0 ** -16 <= m <= v32 + 1e-12
    p = m - np.floor(v32)
    assert var == pytest.approx(p * (1 - p), abs=1e-12)
    assert var <= 0.25 + 1e-12
    if v32 == np.floor(v32):
        assert m == v32 and var == 0.0


def test_sr_takes_only_floor_or_ceil():
    rs = np.random.Generator(np.random.Philox(3))
    for v in rs.uniform(0, 31, 200).astype(np.float32):
        for u in (0, 1, 12345, 40000, 65535):
            c = orc.sr(v, u, 31)
            assert c in (np.floor(v), min(np.ceil(v), 31))


# --------------------------------------------------------------------------
# Unbiasedness of every quantizer, exactly (enumerating all outcomes)
# --------------------------------------------------------------------------
CASES = [(orc.PTQ, 4, 0), (orc.PTQ, 8, 0), (orc.PSQ, 3, 0), (orc.PSQ, 8, 0),
         (orc.BHQ, 4, 4), (orc.BHQ, 5, 3), (orc.BHQ, 8, 8), (orc.BHQ, 2, 1)]


@pytest.mark.parametrize("kind,bits,block", CASES)
def test_quantizer_is_unbiased_exactly(kind, bits, block):
    g = wl.rng(11 + kind * 10 + bits)
    h = wl.random_grad(g, 8, 12, sigma=2.0, outlier_frac=0.2)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, kind, bits, block, seed=5, want_v=True)
    v = q["v"]
    assert v.min() >= 0.0 and v.max() <= B * (1 + 1e-5)
    m, _ = _moments(v, B)
    e_deq = orc.dequant(q, m)
    nb = block if kind == orc.BHQ else (1 if kind == orc.PSQ else 8)
    for r0, n in _blocks(8, nb):
        scale = np.abs(h[r0:r0 + n]).max()
        err = np.abs(e_deq[r0:r0 + n] - h[r0:r0 + n]).max()
        assert err <= 2e-5 * scale, (r0, err, scale)


# --------------------------------------------------------------------------
# Exact variance against the paper's expressions
# --------------------------------------------------------------------------
def _exact_var_of_dequant(q, var_codes):
    """Var of each dequantized entry: diag(inv_s) Q_blk acts on independent codes."""
    n, c = var_codes.shape
    inv_s = q["inv_s"].astype(np.float64)
    if q["kind"] == orc.PTQ:
        return var_codes * inv_s[0] ** 2
    if q["kind"] == orc.PSQ:
        return var_codes * (inv_s ** 2)[:, None]
    out = np.zeros((n, c))
    for b, (r0, nb) in enumerate(_blocks(n, q["block"])):
        Q = orc.householder(nb, int(q["lead"][b]))
        W = (inv_s[r0:r0 + nb, None] * Q) ** 2
        out[r0:r0 + nb] = W @ var_codes[r0:r0 + nb]
    return out


@pytest.mark.parametrize("bits", [4, 8])
def test_ptq_variance_bound(bits):
    g = wl.rng(21)
    h = wl.random_grad(g, 6, 16)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.PTQ, bits, want_v=True)
    _, var = _moments(q["v"], B)
    total = _exact_var_of_dequant(q, var).sum()
    R = float(h.max() - h.min())
    assert total <= h.size * R * R / (4 * B * B) * (1 + 1e-5)  # Eq. 8
    assert total > 0


@pytest.mark.parametrize("bits", [3, 5])
def test_psq_variance_bound_and_gain(bits):
    g = wl.rng(22)
    h = wl.random_grad(g, 8, 16, sigma=2.0)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.PSQ, bits, want_v=True)
    _, var = _moments(q["v"], B)
    total = _exact_var_of_dequant(q, var).sum()
    Ri = h.max(axis=1) - h.min(axis=1)
    bound = h.shape[1] / (4 * B * B) * (Ri.astype(np.float64) ** 2).sum()
    assert total <= bound * (1 + 1e-5)  # Sec. 4.1 / App. D.3
    qp = orc.quantize_grad(h, orc.PTQ, bits, want_v=True)
    _, varp = _moments(qp["v"], B)
    assert total < _exact_var_of_dequant(qp, varp).sum()  # PSQ below PTQ


@pytest.mark.parametrize("nb,bits", [(4, 4), (8, 5), (16, 8)])
def test_bhq_variance_bound(nb, bits):
    g = wl.rng(23 + nb)
    h = (1e-3 * g.standard_normal((2 * nb, 10))).astype(np.float32)
    h[0] = 10.0 * g.standard_normal(10)
    h[nb + 3] = 30.0 * g.standard_normal(10)
    # one large row per block, lambda2 / lambda1 ~ 0: the case of Sec. 4.2
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.BHQ, bits, nb, want_v=True)
    _, var = _moments(q["v"], B)
    vd = _exact_var_of_dequant(q, var)
    D = h.shape[1]
    for b, (r0, n) in enumerate(_blocks(h.shape[0], nb)):
        blk = h[r0:r0 + n].astype(np.float64)
        p = int(np.argmax(np.abs(blk).max(axis=1)))
        assert p == q["lead"][b]
        lam1 = blk[p].max() - blk[p].min()
        lam2 = 2 * np.delete(np.abs(blk).max(axis=1), p).max()
        inv_s = q["inv_s"][r0:r0 + n].astype(np.float64)
        frob = (inv_s ** 2).sum()  # ||S^-1||_F^2, Q orthogonal
        var_blk = vd[r0:r0 + n].sum()
        assert var_blk <= D / 4 * frob * (1 + 1e-6)  # matrix-quantizer bound
        hh = (lam1 ** (2 / 3) * n ** (-1 / 3) + lam2 ** (2 / 3) * n ** (2 / 3)) ** 3
        assert frob <= hh / B ** 2 * (1 + 1e-5)  # App. D.4
    # in this regime BHQ has lower variance than PSQ (Sec. 4.2)
    qs = orc.quantize_grad(h, orc.PSQ, bits, want_v=True)
    _, vs = _moments(qs["v"], B)
    assert vd.sum() < _exact_var_of_dequant(qs, vs).sum()


def test_fewer_bits_cost_about_4x_variance():
    g = wl.rng(24)
    h = g.standard_normal((16, 32)).astype(np.float32)
    tot = {}
    for bits in (4, 5, 6):
        q = orc.quantize_grad(h, orc.PTQ, bits, want_v=True)
        _, var = _moments(q["v"], (1 << bits) - 1)
        tot[bits] = _exact_var_of_dequant(q, var).sum()
    for b in (5, 6):
        expect = (((1 << b) - 1) / ((1 << (b - 1)) - 1)) ** 2  # Sec. 3.3
        assert tot[b - 1] / tot[b] == pytest.approx(expect, rel=0.2)


# --------------------------------------------------------------------------
# Householder reflection and the BHQ construction (Sec. 4.2, App. D.4)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("nb,p", [(2, 0), (3, 2), (8, 5), (16, 0), (64, 63)])
def test_householder_identities(nb, p):
    Q = orc.householder(nb, p)
    assert np.allclose(Q @ Q.T, np.eye(nb), atol=1e-12)
    assert np.allclose(Q, Q.T, atol=1e-15)
    e = np.zeros(nb)
    e[p] = 1.0
    assert np.allclose(Q @ e, np.ones(nb) / np.sqrt(nb), atol=1e-12)
    x = np.random.Generator(np.random.Philox(nb)).standard_normal(nb)
    assert np.linalg.norm(Q @ x) == pytest.approx(np.linalg.norm(x), rel=1e-12)


def test_householder_single_row_is_identity():
    assert np.array_equal(orc.householder(1, 0), np.eye(1))


@pytest.mark.parametrize("lam1,lam2,nb", [(10.0, 0.1, 16), (1.0, 1.0, 8),
                                           (3.0, 1e-4, 64), (2.0, 0.5, 2)])
def test_bhq_scales_solve_the_constrained_problem(lam1, lam2, nb):
    B = 31
    s1, s2 = orc.bhq_scales(lam1, lam2, nb, B)
    # The range constraint of App. D.4 holds with equality ...
    assert lam1 * s1 / np.sqrt(nb) + lam2 * s2 * np.sqrt(nb) == pytest.approx(B)
    # ... and s1, s2 minimise s1^-2 + N s2^-2 along it.
    f = lambda a: a ** -2 + nb * ((B - lam1 * a / np.sqrt(nb)) / (lam2 * np.sqrt(nb))) ** -2
    for eps in (1e-3, -1e-3):
        assert f(s1 * (1 + eps)) > f(s1)
    # and the objective equals the closed form of App. D.4.
    hh = (lam1 ** (2 / 3) * nb ** (-1 / 3) + lam2 ** (2 / 3) * nb ** (2 / 3)) ** 3
    assert s1 ** -2 + nb * s2 ** -2 == pytest.approx(hh / B ** 2, rel=1e-12)


def test_bhq_range_stays_within_B():
    g = wl.rng(31)
    for trial in range(20):
        nb = [2, 4, 8, 16, 32, 64][trial % 6]
        h = wl.random_grad(g, 4 * nb + 3, 24, sigma=2.5, outlier_frac=0.05)
        for bits in (2, 5, 8):
            q = orc.quantize_grad(h, orc.BHQ, bits, nb, want_v=True)
            B = (1 << bits) - 1
            assert q["v"].min() >= 0.0
            assert q["v"].max() <= B * (1 + 1e-5)


def test_bhq_degenerate_blocks():
    h = np.zeros((12, 8), dtype=np.float32)
    h[4] = 3.0  # constant lead row, lambda1 = 0, lambda2 = 0
    h[9] = np.linspace(-1, 2, 8)  # single live row in its block
    q = orc.quantize_grad(h, orc.BHQ, 5, 4)
    assert (q["codes"][:4] == 0).all() and (q["inv_s"][:4] == 0).all()
    assert q["lead"].tolist() == [0, 0, 1]
    deq = orc.dequant(q)
    assert np.abs(deq - h).max() <= (3.0 / 31) + 1e-6
    assert np.allclose(deq[:4], 0.0)
    # rows that are zero dequantize to zero exactly (inv_s = 0)
    assert (q["inv_s"][[5, 6, 7, 8, 10, 11]] == 0).all()


def test_bhq_block_one_matches_psq():
    g = wl.rng(32)
    h = wl.random_grad(g, 64, 64)
    a = orc.quantize_grad(h, orc.BHQ, 5, 1, seed=9)
    b = orc.quantize_grad(h, orc.PSQ, 5, seed=9)
    diff = a["codes"].astype(int) - b["codes"].astype(int)
    assert (diff == 0).mean() > 0.999 and np.abs(diff).max() <= 1
    assert np.allclose(a["inv_s"], b["inv_s"], rtol=1e-6)


def test_psq_reduces_to_ptq_when_rows_share_a_range():
    g = wl.rng(33)
    base = g.standard_normal(32).astype(np.float32)
    h = np.stack([g.permutation(base) for _ in range(10)])
    a = orc.quantize_grad(h, orc.PSQ, 5, seed=4)
    b = orc.quantize_grad(h, orc.PTQ, 5, seed=4)
    assert np.array_equal(a["codes"], b["codes"])  # S = s I (Eq. 9 remark)
    assert np.all(a["inv_s"] == b["inv_s"][0]) and np.all(a["zero"] == b["zero"][0])


def test_constant_and_zero_rows():
    h = np.zeros((4, 16), dtype=np.float32)
    h[1] = 2.5
    h[2] = np.arange(16)
    for kind in (orc.PTQ, orc.PSQ):
        q = orc.quantize_grad(h, kind, 4)
        deq = orc.dequant(q)
        if kind == orc.PSQ:
            assert np.array_equal(q["codes"][:2], np.zeros((2, 16)))
            assert np.allclose(deq[:2], h[:2])


# --------------------------------------------------------------------------
# Deterministic forward quantizer (Sec. 2.1, App. E)
# --------------------------------------------------------------------------
def test_forward_quantizer_rounds_half_to_even():
    x = np.array([[0.0, 0.5, 1.5, 2.5, 3.5, 254.5, 255.0, 7.49]], dtype=np.float32)
    q = orc.quantize_fwd(x, 8)  # min 0, max 255 -> s = 1
    assert q["inv_s"][0] == 1.0
    assert q["codes"].tolist() == [[0, 0, 2, 2, 4, 254, 255, 7]]


def test_forward_quantizer_error_is_half_a_bin():
    g = wl.rng(34)
    x = g.uniform(-3, 5, (40, 50)).astype(np.float32)
    q = orc.quantize_fwd(x, 8)
    deq = orc.dequant(q)
    assert q["codes"].min() == 0 and q["codes"].max() == 255
    assert np.abs(deq - x).max() <= 0.5 * q["inv_s"][0] * (1 + 1e-4) + 1e-6


# --------------------------------------------------------------------------
# Contractions: integer GEMM and Thm 1
# --------------------------------------------------------------------------
@pytest.mark.parametrize("ak,bk", [(1, 0), (0, 0), (1, 1), (0, 1)])
def test_int_gemm_matches_numpy(ak, bk):
    g = wl.rng(41)
    M, N, K = 7, 9, 33
    A = g.integers(0, 256, (M, K)).astype(np.uint8)
    Bm = g.integers(0, 32, (K, N)).astype(np.uint8)
    a_st = A if ak else A.T.copy()
    b_st = Bm.T.copy() if bk else Bm
    P = orc.int_gemm(a_st, ak, b_st, bk, M, N, K, 128, 16)
    ref = (A.astype(np.int64) - 128) @ (Bm.astype(np.int64) - 16)
    assert np.array_equal(P, ref)


def test_matmul_matches_numpy():
    g = wl.rng(42)
    A = g.standard_normal((5, 7))
    Bm = g.standard_normal((7, 3))
    assert np.allclose(orc.matmul(A, Bm), A @ Bm, rtol=1e-13)
    assert np.allclose(orc.matmul(A.T.copy(), Bm, a_trans=True), A @ Bm, rtol=1e-13)


@pytest.mark.parametrize("kind,bits,block", [(orc.PTQ, 5, 0), (orc.PSQ, 4, 0),
                                             (orc.BHQ, 5, 4), (orc.BHQ, 5, 0)])
def test_fqt_gradients_are_unbiased_exactly(kind, bits, block):
    """Thm 1: E[FQT gradient | batch] = QAT gradient, for both contractions."""
    g = wl.rng(51)
    dH = wl.random_grad(g, 8, 10, outlier_frac=0.25)
    X = g.uniform(-1, 1, (8, 6)).astype(np.float32)
    W = (0.3 * g.standard_normal((10, 6))).astype(np.float32)
    qx, qw = orc.quantize_fwd(X), orc.quantize_fwd(W)
    q2 = orc.quantize_grad(dH, kind, bits, block, want_v=True)
    q1 = orc.quantize_grad(dH, orc.PTQ, 8, 0, stream=orc.STREAM_B1, want_v=True)
    m2, _ = _moments(q2["v"], (1 << bits) - 1)
    m1, _ = _moments(q1["v"], 255)
    Wt, Xt = orc.dequant(qw), orc.dequant(qx)
    e_gx = orc.matmul(orc.dequant(q2, m2), Wt)
    e_gw = orc.matmul(orc.dequant(q1, m1), Xt, a_trans=True)
    qat_gx = dH.astype(np.float64) @ Wt
    qat_gw = dH.astype(np.float64).T @ Xt
    assert np.abs(e_gx - qat_gx).max() <= 1e-4 * np.abs(qat_gx).max()
    assert np.abs(e_gw - qat_gw).max() <= 1e-4 * np.abs(qat_gw).max()
    # and a single draw is what grad_x / grad_w return
    assert np.allclose(orc.grad_x(q2, qw), orc.matmul(orc.dequant(q2), Wt))


@pytest.mark.parametrize("kind,bits,block", [(orc.PSQ, 4, 0), (orc.BHQ, 4, 8)])
def test_monte_carlo_mean_and_variance(kind, bits, block):
    """Over many seeds: per-entry z-scores of the mean, total variance and the
    variance of grad_X (Prop. 3's equality form, independent codes)."""
    g = wl.rng(61)
    h = wl.random_grad(g, 16, 32, outlier_frac=0.1)
    W = (0.5 * g.standard_normal((32, 8))).astype(np.float32)
    B = (1 << bits) - 1
    q0 = orc.quantize_grad(h, kind, bits, block, want_v=True)
    _, var_codes = _moments(q0["v"], B)
    vd = _exact_var_of_dequant(q0, var_codes)
    Wt = orc.dequant(orc.quantize_fwd(W))
    K = 768
    s1 = np.zeros(h.shape)
    s2 = np.zeros(h.shape)
    gx = []
    for seed in range(K):
        q = orc.quantize_grad(h, kind, bits, block, seed=seed + 1000)
        d = orc.dequant(q)
        s1 += d
        s2 += d * d
        gx.append(d @ Wt)
    mean = s1 / K
    emp_var = s2 / K - mean ** 2
    live = vd > 0
    z = (mean - h)[live] / np.sqrt(vd[live] / K)
    assert np.abs(z).max() < 5.5
    assert emp_var.sum() / vd.sum() == pytest.approx(1.0, rel=0.1)
    gx = np.array(gx)
    # exact Var[grad_X] from the independent per-code variances
    n = h.shape[0]
    inv_s = q0["inv_s"].astype(np.float64)
    if kind == orc.PSQ:
        var_gx = ((inv_s ** 2)[:, None] * var_codes) @ (Wt ** 2)
    else:
        var_gx = np.zeros((n, Wt.shape[1]))
        for b, (r0, nbk) in enumerate(_blocks(n, block)):
            Q = orc.householder(nbk, int(q0["lead"][b]))
            A = inv_s[r0:r0 + nbk, None] * Q
            var_gx[r0:r0 + nbk] = (A ** 2) @ (var_codes[r0:r0 + nbk] @ (Wt ** 2))
    assert gx.var(axis=0).sum() / var_gx.sum() == pytest.approx(1.0, rel=0.12)


def test_linear_backward_shapes_and_bifurcation():
    L = wl.config(0, rows=16)[0]
    out = orc.linear_backward(L.dH, L.X, L.W, orc.BHQ, 5, 16, seed=0)
    assert out["grad_x"].shape == (16, 256) and out["grad_w"].shape == (256, 256)
    assert out["q_b1"]["bits"] == 8 and out["q_b1"]["kind"] == orc.PTQ
    # stream 1 draws differ from stream 0 draws
    q2p = orc.quantize_grad(L.dH, orc.PTQ, 8, 0, seed=0, stream=0)
    assert not np.array_equal(q2p["codes"], out["q_b1"]["codes"])


# --------------------------------------------------------------------------
# Adaptive BHQ grouping (App. D.5, reading R8 of the oracle)
# --------------------------------------------------------------------------
def _groups(q):
    """(stored start, size) of every adaptive group."""
    gs = q["gstart"]
    return [(int(gs[i]), int(gs[i + 1] - gs[i])) for i in range(q["G"])]


def test_bhq_grouping_worked_example():
    """N = 4 rows with M = (1, 1, 8, 1).  Per group the estimate is
    (M^(2/3) + L^(2/3) size)^3 / size, so by hand:
    G = 1: size 3, L = 1:            (4 + 3)^3 / 3 = 343 / 3;
    G = 2: sizes 16/9, 2/9, L = 1:   (52/9)^3 (9/16) + (11/9)^3 (9/2)
                                     = 151256 / 1296;
    G = 3: sizes 0.8, 0.1, 0.1:      4.8^3 / 0.8 + 2 (1.1^3 / 0.1) = 164.86.
    G = 1 wins: one group, the row with M = 8 first, then rows 0, 1, 3."""
    h = np.zeros((4, 8), np.float32)
    h[:, 0] = [1, -1, 8, 1]
    h[:, 3] = [0.5, 0.2, -3, 0.1]
    g = orc.bhq_grouping(h, want_v=True)
    assert np.allclose(g["V"], [343 / 3, 151256 / 1296, 164.86], rtol=1e-13, atol=0)
    assert g["G"] == 1
    assert list(g["perm"]) == [2, 0, 1, 3]
    assert list(g["gstart"]) == [0, 4, 4, 4, 4]
    assert list(g["gsize"]) == [4, 4, 4, 4]


@pytest.mark.parametrize("n", [2, 10, 11, 64])
def test_bhq_grouping_equal_rows(n):
    """All M_i = c: size = (N - G) / G and V(G) = c^2 N^3 / (G (N - G)),
    smallest at G = N / 2 (symmetric about it), i.e. pairs for even N; the
    small rows are dealt from the end of the index order."""
    c = 1.75
    h = np.zeros((n, 16), np.float32)
    h[:, 5] = c
    h[1::2, 5] = -c
    g = orc.bhq_grouping(h, want_v=True)
    G = np.arange(1, n)
    assert np.allclose(g["V"], c * c * n ** 3 / (G * (n - G)), rtol=1e-12, atol=0)
    if n % 2 == 0:
        assert g["G"] == n // 2
        perm = g["perm"].reshape(-1, 2)
        assert np.array_equal(perm[:, 0], np.arange(n // 2))
        assert np.array_equal(perm[:, 1], n - 1 - np.arange(n // 2))
        assert np.all(g["gsize"] == 2)
    else:
        assert g["G"] in ((n - 1) // 2, (n + 1) // 2)


def test_bhq_grouping_small_rows_vanish():
    """With the small rows all zero (L = 0) the estimate is App. D.5's own
    sum_i M_i^2 / size_i = (sum_{i<=G} M_i)^2 / (N - G)."""
    g0 = wl.rng(71)
    n, K = 40, 6
    h = np.zeros((n, 24), np.float32)
    rows = g0.choice(n, K, replace=False)
    h[rows] = g0.standard_normal((K, 24)) * np.array([9, 5, 3, 2, 1.5, 1.2])[:, None]
    M = np.sort(np.abs(h).max(axis=1).astype(np.float64))[::-1]
    g = orc.bhq_grouping(h, want_v=True)
    for G in range(K, n):
        assert g["V"][G - 1] == pytest.approx(M[:K].sum() ** 2 / (n - G), rel=1e-12)
    assert g["G"] <= K
    assert set(g["perm"][g["gstart"][:g["G"]]]) == set(rows[np.argsort(
        -np.abs(h[rows]).max(axis=1))][:g["G"]])


@pytest.mark.parametrize("n,seed", [(1, 0), (3, 1), (37, 2), (128, 3), (500, 4)])
def test_bhq_grouping_invariants(n, seed):
    """Partition, leads = the G largest rows, cumulative-rounding sizes within
    one row of (N - G) M_i / S_G, small rows dealt from the smallest up, and
    V(G) equal to its expansion in prefix sums of M^(1), M^(4/3), M^(5/3),
    M^2 (term = M (t + M^(1/3) u)^3, t = (S_G / (N - G))^(1/3),
    u = L^(2/3) ((N - G) / S_G)^(2/3))."""
    g0 = wl.rng(80 + seed)
    h = wl.random_grad(g0, n, 16, sigma=2.0, outlier_frac=0.05)
    g = orc.bhq_grouping(h, want_v=True)
    G, perm, gs = g["G"], g["perm"], g["gstart"]
    assert np.array_equal(np.sort(perm), np.arange(n))
    assert gs[0] == 0 and np.all(np.diff(gs[:G + 1]) >= 1) and np.all(gs[G:] == n)
    M = np.abs(h).max(axis=1).astype(np.float64)
    order = np.lexsort((np.arange(n), -M))
    assert np.array_equal(perm[gs[:G]], order[:G])
    if n == 1:
        assert G == 1
        return
    Ms = M[order]
    SG = Ms[:G].sum()
    sizes = np.diff(gs[:G + 1]) - 1
    assert sizes.sum() == n - G
    assert np.all(np.abs(sizes - (n - G) * Ms[:G] / SG) <= 1.0 + 1e-9)
    for i, (k0, nb) in enumerate(_groups(g)):
        assert np.all(g["gsize"][k0:k0 + nb] == nb)
        assert np.all(M[perm[k0 + 1:k0 + nb]] <= M[perm[k0]])
        if i + 1 < G and nb > 1 and gs[i + 2] - gs[i + 1] > 1:
            assert M[perm[k0 + 1:k0 + nb]].max() <= M[perm[gs[i + 1] + 1:gs[i + 2]]].min()
    Gs = np.arange(1, n)
    S = np.cumsum(Ms)[:-1]
    t = (S / (n - Gs)) ** (1 / 3)
    u = Ms[1:] ** (2 / 3) * ((n - Gs) / S) ** (2 / 3)
    P = [np.cumsum(Ms ** e)[:-1] for e in (1.0, 4 / 3, 5 / 3, 2.0)]
    V = t ** 3 * P[0] + 3 * t ** 2 * u * P[1] + 3 * t * u ** 2 * P[2] + u ** 3 * P[3]
    assert np.allclose(g["V"], V, rtol=1e-10, atol=0)
    assert g["V"][G - 1] == g["V"].min() and np.argmin(g["V"]) == G - 1


def test_bhq_adaptive_single_group_is_the_blocked_bhq():
    """One group in index order is the contiguous BHQ with block = N: same
    codes, scales and zero points bit for bit."""
    n = 8
    h = np.zeros((n, 16), np.float32)
    g0 = wl.rng(90)
    h[0] = 40.0 * g0.standard_normal(16)
    for k in range(1, n):
        h[k] = g0.uniform(-0.5, 0.5, 16)
        h[k, k] = 1.0 - 0.01 * k  # strictly decreasing M in index order
    q = orc.quantize_grad(h, orc.BHQ, 5, 0, seed=4, want_v=True)
    assert q["G"] == 1 and np.array_equal(q["perm"], np.arange(n))
    r = orc.quantize_grad(h, orc.BHQ, 5, n, seed=4, want_v=True)
    assert r["lead"][0] == 0
    for key in ("codes", "inv_s", "zero", "v"):
        assert np.array_equal(q[key], r[key]), key
    assert np.array_equal(orc.dequant(q), orc.dequant(r))


@pytest.mark.parametrize("bits,n", [(4, 12), (5, 9), (8, 16)])
def test_bhq_adaptive_is_unbiased_exactly(bits, n):
    g0 = wl.rng(100 + bits)
    h = wl.random_grad(g0, n, 10, sigma=2.0, outlier_frac=0.2)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.BHQ, bits, 0, seed=5, want_v=True)
    v = q["v"]
    assert v.min() >= 0.0 and v.max() <= B * (1 + 1e-5)
    m, _ = _moments(v, B)
    e_deq = orc.dequant(q, m)
    for k0, nb in _groups(q):
        rows = q["perm"][k0:k0 + nb]
        scale = np.abs(h[rows]).max()
        assert np.abs(e_deq[rows] - h[rows]).max() <= 2e-5 * scale


@pytest.mark.parametrize("bits", [4, 6])
def test_bhq_adaptive_variance_bound(bits):
    """Per adaptive group: exact variance <= D/4 ||S^-1||_F^2 and
    ||S^-1||_F^2 <= App. D.4's bound with that group's lambda1, lambda2, n."""
    g0 = wl.rng(110 + bits)
    h = (1e-2 * g0.standard_normal((24, 10))).astype(np.float32)
    h[3] = 10.0 * g0.standard_normal(10)
    h[17] = 25.0 * g0.standard_normal(10)
    h[9] = 4.0 * g0.standard_normal(10)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.BHQ, bits, 0, want_v=True)
    _, var = _moments(q["v"], B)
    D = h.shape[1]
    assert q["G"] >= 2
    for k0, nb in _groups(q):
        rows = q["perm"][k0:k0 + nb]
        inv_s = q["inv_s"][k0:k0 + nb].astype(np.float64)
        Q = orc.householder(nb, 0)
        vd = ((inv_s[:, None] * Q) ** 2) @ var[k0:k0 + nb]
        frob = (inv_s ** 2).sum()
        assert vd.sum() <= D / 4 * frob * (1 + 1e-6)
        if nb > 1:
            blk = h[rows].astype(np.float64)
            lam1 = blk[0].max() - blk[0].min()
            lam2 = 2 * np.abs(blk[1:]).max()
            hh = (lam1 ** (2 / 3) * nb ** (-1 / 3) + lam2 ** (2 / 3) * nb ** (2 / 3)) ** 3
            assert frob <= hh / B ** 2 * (1 + 1e-5)


# --------------------------------------------------------------------------
# Per-sample power-of-two shift quantizer (Sec. 4.3, reading R9 of the oracle)
# --------------------------------------------------------------------------
def test_shift_quantizer_shift_values():
    """Rows scaled by known powers of two: shift_i is the largest integer in
    [0, 4] with 2^shift ||h_i||_inf <= M (equality allowed), capped at 4."""
    base = np.linspace(-1.0, 1.0, 16, dtype=np.float32)  # ||.||_inf = 1
    scales = [1.0, 0.5, 0.5 * 0.999, 0.25, 0.125, 1 / 16, 1 / 64, 0.0, 0.75]
    want = [0, 1, 1, 2, 3, 4, 4, 4, 0]
    h = np.stack([base * np.float32(a) for a in scales]).astype(np.float32)
    q = orc.quantize_grad(h, orc.SHIFT, 5, 0, seed=1)
    assert list(q["shift"]) == want
    s = np.float32(15) / np.float32(1.0)  # (2^(b-1) - 1) / M
    assert np.array_equal(q["inv_s"], np.float32(1) / s * np.float32(2.0) ** -np.array(want, np.float32))
    assert np.all(q["zero"] == -16)


@pytest.mark.parametrize("bits", [3, 5, 8])
def test_shift_quantizer_is_unbiased_exactly_and_in_range(bits):
    g = wl.rng(120 + bits)
    h = wl.random_grad(g, 10, 12, sigma=2.0, outlier_frac=0.2)
    B = (1 << bits) - 1
    q = orc.quantize_grad(h, orc.SHIFT, bits, 0, seed=7, want_v=True)
    v = q["v"]
    assert v.min() >= 1.0 - 1e-5 and v.max() <= B + 1e-5  # |s 2^sh h| <= 2^(b-1) - 1
    m, var = _moments(v, B)
    e = orc.dequant(q, m)
    # E[code] falls below v by less than 2^-16 of a bin (R1), v is fp32
    inv = q["inv_s"].astype(np.float64)[:, None]
    assert np.all(np.abs(e - h) <= inv * 2.0 ** -15)
    # per-entry variance p(1-p) / (s 2^sh)^2 <= 1 / (4 (s 2^sh)^2)
    assert np.all(var * inv ** 2 <= 0.25 * inv ** 2 * (1 + 1e-9))


def test_shift_quantizer_beats_the_symmetric_per_tensor_range():
    """Rows far below the largest get up to 16x finer steps: the exact
    variance falls below the unshifted (shift 0) quantizer's, by up to 256x per
    such row (Sec. 4.3's motivation, Sec. 4.1's per-sample argument)."""
    g = wl.rng(130)
    h = (0.01 * g.standard_normal((8, 16))).astype(np.float32)
    h[2] = 5.0 * g.standard_normal(16)
    bits = 4
    q = orc.quantize_grad(h, orc.SHIFT, bits, 0, want_v=True)
    _, var = _moments(q["v"], (1 << bits) - 1)
    vq = var * (q["inv_s"].astype(np.float64) ** 2)[:, None]
    assert q["shift"][2] == 0 and np.all(np.delete(q["shift"], 2) == 4)
    # the same rows with every shift forced to 0: step 1/s instead of 1/(16 s)
    step0 = q["inv_s"][2].astype(np.float64)
    small = np.delete(np.arange(8), 2)
    assert vq[small].sum() <= small.size * 16 * 0.25 * (step0 / 16) ** 2 * (1 + 1e-9)
    assert vq[small].max() < 0.25 * step0 ** 2 / 200


def test_shift_quantizer_equal_rows_is_symmetric_ptq():
    g = wl.rng(131)
    base = g.standard_normal(16).astype(np.float32)
    h = np.stack([base if k % 2 else -base for k in range(6)])
    q = orc.quantize_grad(h, orc.SHIFT, 6, 0, seed=2)
    assert np.all(q["shift"] == 0)
    assert np.all(q["inv_s"] == q["inv_s"][0])


@pytest.mark.parametrize("bits", [4, 8])
def test_shifted_accumulators_equal_the_dequantized_product(bits):
    """Sec. 4.3's hardware form: integer products of each sample shifted by
    2^(4 - shift_i) before the sum over samples, one scale at the end, equals
    grad_W of the dequantized codes (Eq. 6) up to double rounding."""
    g = wl.rng(140 + bits)
    dH = wl.random_grad(g, 40, 16, sigma=2.5, outlier_frac=0.1)
    X = g.uniform(-1, 1, (40, 24)).astype(np.float32)
    q = orc.quantize_grad(dH, orc.SHIFT, bits, 0, seed=9)
    qx = orc.quantize_fwd(X)
    a = orc.shifted_codes(q)
    assert np.abs(a).max() <= 16 * ((1 << (bits - 1)) - 1)  # fits an fp16 carrier exactly
    ref = orc.grad_w(q, qx)
    got = orc.grad_w_shifted(q, qx)
    assert np.abs(got - ref).max() <= 1e-12 * np.abs(ref).max()


def test_shift_gradients_are_unbiased_exactly():
    """Thm 1 with the shift quantizer feeding both contractions (no
    bifurcation): E[grad_X] and E[grad_W] equal the QAT gradients."""
    g = wl.rng(150)
    dH = wl.random_grad(g, 8, 10, outlier_frac=0.25)
    X = g.uniform(-1, 1, (8, 6)).astype(np.float32)
    W = (0.3 * g.standard_normal((10, 6))).astype(np.float32)
    qx, qw = orc.quantize_fwd(X), orc.quantize_fwd(W)
    q = orc.quantize_grad(dH, orc.SHIFT, 4, 0, want_v=True)
    m, _ = _moments(q["v"], 15)
    Wt, Xt = orc.dequant(qw), orc.dequant(qx)
    e = orc.dequant(q, m)
    assert np.abs(orc.matmul(e, Wt) - dH.astype(np.float64) @ Wt).max() <= 1e-4 * np.abs(dH @ Wt).max()
    assert np.abs(orc.matmul(e, Xt, a_trans=True) - dH.astype(np.float64).T @ Xt).max() <= \
        1e-4 * np.abs(dH.T @ Xt).max()


# --------------------------------------------------------------------------
# Per-image samples and col2im (Sec. 2.1 conv as a linear layer on im2col
# rows; Sec. 4.1 a sample is one input's gradient)
# --------------------------------------------------------------------------
@pytest.mark.parametrize("n,h,w,c,k,stride,pad", [(2, 5, 6, 3, 3, 1, 1), (1, 7, 7, 4, 1, 1, 0),
                                                  (2, 6, 5, 2, 3, 1, 0), (1, 9, 8, 3, 5, 1, 2),
                                                  (2, 8, 8, 3, 3, 2, 1)])
def test_col2im_is_the_adjoint_of_im2col(n, h, w, c, k, stride, pad):
    """<col2im(G), x> = <G, im2col(x)> for every G and x, with the im2col of
    the workload generator (an independent numpy implementation)."""
    g = wl.rng(n * 100 + h * 10 + k)
    x = g.standard_normal((n, h, w, c))
    X = wl.im2col_nhwc(x, k, k, stride, pad)
    G = g.standard_normal(X.shape)
    lhs = float((orc.col2im_nhwc(G, n, h, w, c, k, k, stride, pad) * x).sum())
    rhs = float((G * X).sum())
    assert lhs == pytest.approx(rhs, rel=1e-12, abs=1e-12)


def test_col2im_of_a_one_by_one_conv_is_the_identity():
    g = wl.rng(77)
    G = g.standard_normal((2 * 4 * 5, 3))
    out = orc.col2im_nhwc(G, 2, 4, 5, 3, 1, 1, 1, 0)
    assert np.array_equal(out.reshape(-1, 3), G)


def test_grad_x_nhwc_is_the_transposed_convolution():
    """The input gradient of a stride-1 conv by brute force: dX[n,y,x,ci] =
    sum over taps and output channels of dY[n, y+pad-ky, x+pad-kx, co]
    W[co, ky, kx, ci], against col2im of the dequantized product."""
    g = wl.rng(91)
    n, h, w, ci, co, k, pad = 2, 5, 4, 3, 4, 3, 1
    dH = g.standard_normal((n * h * w, co)).astype(np.float32)
    W = (0.3 * g.standard_normal((co, k * k * ci))).astype(np.float32)
    q2 = orc.quantize_grad_samples(dH, h * w, orc.PSQ, 8, 0, seed=3)
    qw = orc.quantize_fwd(W, 8)
    got = orc.grad_x_nhwc(q2, qw, n, h, w, ci, k, pad)
    dY = orc.dequant_samples(q2).reshape(n, h, w, co)
    Wd = orc.dequant(qw).reshape(co, k, k, ci)
    ref = np.zeros((n, h, w, ci))
    for b in range(n):
        for y in range(h):
            for x in range(w):
                for ky in range(k):
                    for kx in range(k):
                        oy, ox = y + pad - ky, x + pad - kx
                        if 0 <= oy < h and 0 <= ox < w:
                            ref[b, y, x] += dY[b, oy, ox] @ Wd[:, ky, kx]
    assert np.abs(got - ref).max() <= 1e-12 * np.abs(ref).max()


@pytest.mark.parametrize("kind,bits", [(orc.PSQ, 8), (orc.PSQ, 5), (orc.PTQ, 5)])
def test_one_row_samples_are_the_row_quantizer(kind, bits):
    g = wl.rng(5)
    dH = wl.random_grad(g, 12, 16, outlier_frac=0.2)
    a = orc.quantize_grad_samples(dH, 1, kind, bits, 0, seed=9)
    b = orc.quantize_grad(dH, kind, bits, 0, seed=9)
    assert np.array_equal(a["codes"], b["codes"])
    assert np.array_equal(a["inv_s"], b["inv_s"]) and np.array_equal(a["zero"], b["zero"])


def test_per_sample_scale_spans_the_whole_sample():
    """PSQ with samples of R rows: one scale per sample, B / R(h_i) over all
    R C entries of the sample (Sec. 4.1), shared by its rows."""
    g = wl.rng(6)
    R, n, c, bits = 6, 24, 8, 5
    dH = wl.random_grad(g, n, c, sigma=1.5)
    q = orc.quantize_grad_samples(dH, R, orc.PSQ, bits, 0, seed=2)
    B = (1 << bits) - 1
    for i in range(n // R):
        blk = dH[i * R:(i + 1) * R].astype(np.float32)
        rng_ = np.float32(blk.max()) - np.float32(blk.min())
        s = np.float32(B) / rng_
        assert q["inv_s"][i] == np.float32(1.0) / s
        assert np.all(q["inv_s_rows"][i * R:(i + 1) * R] == q["inv_s"][i])
        assert q["codes"][i * R:(i + 1) * R].min() == 0  # the sample's minimum maps to 0
    assert q["codes"].max() <= B


@pytest.mark.parametrize("kind,bits,block", [(orc.PSQ, 5, 0), (orc.PSQ, 8, 0),
                                             (orc.BHQ, 5, 2)])
def test_per_sample_quantizer_is_unbiased_exactly(kind, bits, block):
    g = wl.rng(31 + bits)
    R = 3
    dH = wl.random_grad(g, 12, 4, sigma=2.0, outlier_frac=0.3)
    q = orc.quantize_grad_samples(dH, R, kind, bits, block, seed=4, want_v=True)
    m, _ = _moments(q["v"], (1 << bits) - 1)
    e_deq = orc.dequant_samples(dict(q, codes=m))
    scale = np.abs(dH).max()
    assert np.abs(e_deq - dH).max() <= 2e-5 * scale
