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
