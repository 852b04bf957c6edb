"""Shared helpers of the GPU parity tests (comparison rules of the oracle)."""
import numpy as np
import torch

import oracle as orc


def to_dev(x: np.ndarray, dtype: str = "f32") -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32))
    if dtype == "bf16":
        t = t.to(torch.bfloat16)
    return t.cuda()


def grad_rel_err(g: np.ndarray, r: np.ndarray) -> float:
    """max_ij |g - r| / max(|r_ij|, 1e-3 ||r_i||_inf) (row-relative floor)."""
    r = np.asarray(r, dtype=np.float64)
    g = np.asarray(g, dtype=np.float64)
    floor = 1e-3 * np.abs(r).max(axis=1, keepdims=True)
    den = np.maximum(np.abs(r), floor)
    den = np.where(den > 0, den, 1.0)
    return float((np.abs(g - r) / den).max())


def sr_boundary_distance(v: np.ndarray, seed: int, stream: int, flat_idx):
    """Distance, in units of 2^-16 of a bin, between the fixed-point value of
    v and the stochastic-rounding threshold set by its uniform."""
    out = []
    for vv, i in zip(v, flat_idx):
        u = orc.u16(seed, stream, int(i))
        fixed = int(np.float32(vv) * np.float32(65536.0))
        frac = fixed & 0xFFFF
        out.append(abs((frac + u) - 65536))
    return np.array(out)


def oracle_rows_grad_x(q2: dict, qw: dict, codes2: np.ndarray, rows: np.ndarray):
    """Oracle grad_X restricted to whole quantizer blocks containing `rows`."""
    block = q2["block"] if q2["kind"] == orc.BHQ else 1
    n = codes2.shape[0]
    blocks = sorted(set(int(r) // block for r in rows))
    Wt = orc.dequant(qw)
    out = {}
    for b in blocks:
        r0, r1 = b * block, min(n, (b + 1) * block)
        sub = dict(q2)
        sub["codes"] = codes2[r0:r1]
        if q2["kind"] != orc.PTQ:
            sub["inv_s"] = q2["inv_s"][r0:r1]
            sub["zero"] = q2["zero"][r0:r1]
        if q2["kind"] == orc.BHQ:
            sub["lead"] = q2["lead"][b:b + 1]
        deq = orc.dequant(sub)
        res = orc.matmul(deq, Wt)
        for k in range(r1 - r0):
            out[r0 + k] = res[k]
    return np.stack([out[int(r)] for r in rows])


def oracle_groups_grad_x(q2: dict, qw: dict, groups) -> dict:
    """Oracle grad_X of whole adaptive BHQ groups (stored-order group ids),
    keyed by dH row: each group dequantized on its own (App. D.5 groups are
    independent) and multiplied by W~."""
    Wt = orc.dequant(qw)
    gs = q2["gstart"]
    out = {}
    for gi in groups:
        k0, k1 = int(gs[gi]), int(gs[gi + 1])
        nb = k1 - k0
        sub = dict(q2)
        sub.update(codes=q2["codes"][k0:k1], inv_s=q2["inv_s"][k0:k1],
                   zero=q2["zero"][k0:k1], perm=np.arange(nb, dtype=np.int32),
                   gstart=np.array([0, nb], dtype=np.int32), G=1)
        res = orc.matmul(orc.dequant(sub), Wt)
        for r in range(nb):
            out[int(q2["perm"][k0 + r])] = res[r]
    return out


def grouping_closed_form(dH: np.ndarray):
    """App. D.5 grouping estimate V(G) for every G, from prefix sums of the
    sorted M^p (the expansion of the per-group cube), and the cumulative-
    rounding small-row counts e_i for a given G.  Independent of the oracle's
    direct per-G loop; used where that loop is too slow (large N)."""
    M = np.abs(dH).max(axis=1).astype(np.float32).astype(np.float64)
    n = M.size
    order = np.lexsort((np.arange(n), -M))
    Ms = M[order]
    G = np.arange(1, n)
    S = np.cumsum(Ms)
    P = [np.cumsum(Ms ** e)[:-1] for e in (1.0, 4 / 3, 5 / 3, 2.0)]
    with np.errstate(divide="ignore", invalid="ignore"):
        t = (P[0] / (n - G)) ** (1 / 3)
        u = Ms[1:] ** (2 / 3) * ((n - G) / P[0]) ** (2 / 3)
        V = t ** 3 * P[0] + 3 * t ** 2 * u * P[1] + 3 * t * u ** 2 * P[2] + u ** 3 * P[3]
    V = np.where(P[0] > 0, V, 0.0)

    def sizes(g):
        SG = S[g - 1]
        e = np.zeros(g + 1, dtype=np.int64)
        if SG > 0:
            e[1:g] = np.floor((n - g) * (S[:g - 1] / SG) + 0.5)
        e[g] = n - g
        return e
    return order, Ms, V, sizes
