"""Benchmark of the FQT quantized backward on GB300.

One step = one pass of the whole hot path over the full ResNet-50 v1.5
backward at batch 256, 224 x 224 (53 convolutions and the fc, each lowered to
im2col; 4.19 TOP of integer contractions):  for every layer
  X~ = Q_f(X), W~ = Q_theta(W)            (deterministic 8-bit PTQ)
  Q_b2(dH) = BHQ 5-bit, block 16; Q_b1(dH) = 8-bit stochastic PTQ
  grad_X = Q_b2(dH) W~,  grad_W = Q_b1(dH)^T X~
The reported value is quantized-backward throughput in TOPS: both
contractions count 2 N C D integer ops each.  The stride-1 3 x 3 convolutions
(13 of them) are lowered to their implicit im2col matrix: X stays the NHWC
input, Q_f reads it once and grad_W reads the codes at each tap's offset (the
codes, the contractions and the gradients are those of the explicit im2col
matrix, bit for bit).  Every layer's inputs (fp32 dH, X, W) are resident in
HBM when timing starts; a step moves far more than the 129 MB L2, so no flush
is needed between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

The reference arm times the CPU oracle on a bounded sample of the same
workload (every layer at batch 1) on all host cores.  The other workloads
(the linear layer, the ResNet-18 and ResNet-50 layer3 convs, the transformer
FFN pair) and the method's variants are reported as extras.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "quantized-backward TOPS and quantizer GB/s (1 GB300) vs roofline, oracle-exact"
WORKLOAD = ("resnet50-sweep-b256-224x224: ResNet-50 v1.5 backward, batch 256, 53 convs + fc "
            "via im2col (stem D 147 -> 160, fc C 1000 -> 1008 zero-padded)")
KIND, BITS, BLOCK = 2, 5, 16  # Q_b2 = BHQ-5, block 16
SWEEP_BATCH = 256
CALLS = ["quantize_act", "quantize_weight", "quantize_grad", "grad_x", "grad_w"]
KERNELS = {"quantize_act": "k_range + k_fwd_codes", "quantize_weight": "k_range + k_fwd_codes",
           "quantize_grad": "k_bhq_stats + k_bhq_codes + k_bhq_offsets", "grad_x": "k_gemm",
           "grad_w": "split-K k_gemm + k_reduce"}


def _peaks():
    """(HBM GB/s, bf16 dense TFLOP/s burst, source)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


def _traffic_record(kernel: str, workload: str):
    """Per-launch DRAM bytes of `kernel` on `workload` from the committed ncu
    summary, if that summary was taken on the current kernel sources."""
    path = os.path.join(ROOT, "profiles", "dram_traffic.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    import hashlib
    src = os.path.join(ROOT, "paper_2010_14298_gb300", "csrc")
    h = hashlib.sha256()
    for f in sorted(os.listdir(src)):
        h.update(open(os.path.join(src, f), "rb").read())
    digest = h.hexdigest()[:16]
    for line in text.splitlines():
        parts = [p.strip() for p in line.strip().strip("|").split("|")]
        if len(parts) >= 4 and parts[0] == kernel and parts[1] == workload and parts[3] == digest:
            try:
                return float(parts[2])
            except ValueError:
                return None
    return None


class Clocks:
    """Samples SM clocks and throttle reasons with nvidia-smi while running.

    A reader thread stamps every sample with the host clock on arrival, so
    the summary keeps only samples taken between mark_start() and
    mark_end() (the timed region).  nvidia-smi is started before the region
    and the caller waits for its first sample before starting the clock.
    """
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]

    def __init__(self, index: int, period_ms: int = 50):
        self.index = index
        self.period_ms = period_ms
        self.proc = None
        self.rows = []  # (host time, fields)
        self.t0 = self.t1 = None
        self._thread = None

    def _reader(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 9:
                self.rows.append((time.perf_counter(), parts))

    def __enter__(self):
        import threading
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", str(self.period_ms)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True, bufsize=1)
            self._thread = threading.Thread(target=self._reader, daemon=True)
            self._thread.start()
        except Exception:
            self.proc = None
        return self

    def wait_first(self, timeout_s: float = 10.0):
        t = time.perf_counter()
        while self.proc is not None and not self.rows and time.perf_counter() - t < timeout_s:
            time.sleep(0.01)

    def mark_start(self):
        self.t0 = time.perf_counter()

    def mark_end(self):
        self.t1 = time.perf_counter()

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            if self._thread is not None:
                self._thread.join(timeout=2)

    def summary(self):
        if self.proc is None or not self.rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        t0 = self.t0 if self.t0 is not None else -1e30
        t1 = self.t1 if self.t1 is not None else 1e30
        inside = [r for t, r in self.rows if t0 <= t <= t1]
        where = "timed region"
        if not inside:  # region shorter than one period: the nearest sample after its start
            after = [r for t, r in self.rows if t >= t0]
            inside = after[:1] or [self.rows[-1][1]]
            where = "first sample after the start of the timed region"
        num = lambda v: v.replace(".", "", 1).isdigit()
        sm = [float(r[1]) for r in inside if num(r[1])]
        mx = [float(r[2]) for r in inside if num(r[2])]
        pw = [float(r[3]) for r in inside if num(r[3])]
        reasons = sorted({self.NAMES[i] for r in inside for i in range(4)
                          if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "power_w": statistics.median(pw) if pw else None,
                "samples": len(inside), "sampled": where}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def rank_seed(rank: int, layer: int) -> int:
    """Seed of a rank's synthetic layer: replicas process independent batches
    of the same shapes and distributions (weak scaling)."""
    return 1234 + 4 + layer + 1000 * rank


def max_over_ranks(value: float, device) -> float:
    """The job's time is the slowest rank's: MAX all-reduce of one float
    (the only collective; none is on the data path)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# Algorithmic work per call: each input read once, each output written once,
# codes at 1 byte each, per-row / per-column metadata at 4 bytes per entry.
# (The library's contractions read 2-byte fp16 carriers of the codes; the
# carriers, a PTQ range pass's second read of its input and any re-read from
# L2 are traffic, not algorithmic bytes.)
# ---------------------------------------------------------------------------
def alg_bytes(N: int, C: int, D: int, eb: int = 4, block: int = BLOCK) -> dict:
    nblk = (N + block - 1) // block if block else 0
    return {
        "quantize_act": N * D * eb + N * D + D * 4 + 8,
        "quantize_weight": C * D * eb + C * D + D * 4 + 8,
        "quantize_grad": N * C * eb + 2 * N * C + N * 20 + nblk * 4 + C * 4 + 8,
        "grad_x": N * C + C * D + N * D * 4 + N * 12 + nblk * 4 + D * 4,
        "grad_w": N * C + N * D + C * D * 4 + (C + D) * 4,
    }


def launches(C: int, kind: int = KIND, block: int = BLOCK, implicit: bool = False) -> dict:
    """Kernels each call launches (fixed by the library's dispatch): Q_f and
    Q_theta are a range pass and a code pass; the fixed-block BHQ quantizer on
    the widths of its two-pass form is a statistics pass, a code pass and the
    grad_X offsets, on other widths a range pass, one fused pass and the
    offsets (PTQ and PSQ: a range pass and one fused pass); grad_X is one
    contraction, grad_W the split-K contraction and its reduction; an
    implicit im2col X~ adds the column sums to Q_f and the padding sums to
    grad_W."""
    return {"quantize_act": 3 if implicit else 2, "quantize_weight": 2,
            "quantize_grad": 3 if kind == KIND else 2,
            "grad_x": 1, "grad_w": 3 if implicit else 2}


def implicit_ok(sh) -> bool:
    """A stride-1 3 x 3 conv whose grad_W reads the implicit im2col X~ (the
    NHWC input, read once by Q_f) in blocks of whole output rows."""
    ow = sh.hout
    return (sh.k == 3 and sh.stride == 1 and sh.pad == 1 and sh.cin % 64 == 0 and
            sh.D_pad == sh.D and (ow <= 64 or ow % 32 == 0))


def sweep_layer_tensors(sh, batch: int, seed: int, dev, implicit: bool = False):
    """One layer of the sweep drawn on the device with torch's seeded
    generator: the recipe of workloads.resnet50_layer (input U[-1, 1] at the
    layer's input shape lowered by im2col, dH N(0, 1) rows scaled by
    lognormal(0, 2), W N(0, 2 / D); D and C zero-padded to multiples of 16).
    implicit: X is the NHWC input itself (its im2col matrix is the operand,
    never formed)."""
    import torch
    import torch.nn.functional as F
    gen = torch.Generator(device=dev)
    gen.manual_seed(seed)
    Ns, Dp, Cp = sh.rows(batch), sh.D_pad, sh.C_pad
    if implicit:
        x = torch.rand((batch, sh.cin, sh.h, sh.h), generator=gen, device=dev) * 2.0 - 1.0
        X = x.permute(0, 2, 3, 1).contiguous()
        del x
        dH = torch.zeros((Ns, Cp), dtype=torch.float32, device=dev)
        dH[:, :sh.cout] = (torch.randn((Ns, sh.cout), generator=gen, device=dev)
                           * torch.exp(2.0 * torch.randn((Ns, 1), generator=gen, device=dev)))
        W = torch.zeros((Cp, Dp), dtype=torch.float32, device=dev)
        W[:sh.cout, :sh.D] = (torch.randn((sh.cout, sh.D), generator=gen, device=dev)
                              * float(np.sqrt(2.0 / sh.D)))
        return dH, X, W
    X = torch.zeros((Ns, Dp), dtype=torch.float32, device=dev)
    # im2col in slices of the batch (the unfolded tensor of a whole layer can
    # exceed 2 GB)
    per = max(1, batch // 8)
    r0 = 0
    for b0 in range(0, batch, per):
        nb = min(per, batch - b0)
        x = torch.rand((nb, sh.cin, sh.h, sh.h), generator=gen, device=dev) * 2.0 - 1.0
        cols = F.unfold(x, sh.k, padding=sh.pad, stride=sh.stride)
        rows = nb * sh.hout * sh.hout
        X[r0:r0 + rows, :sh.D] = (cols.view(nb, sh.cin, sh.k * sh.k, -1).permute(0, 3, 2, 1)
                                  .reshape(rows, sh.D))
        r0 += rows
        del x, cols
    dH = torch.zeros((Ns, Cp), dtype=torch.float32, device=dev)
    dH[:, :sh.cout] = (torch.randn((Ns, sh.cout), generator=gen, device=dev)
                       * torch.exp(2.0 * torch.randn((Ns, 1), generator=gen, device=dev)))
    W = torch.zeros((Cp, Dp), dtype=torch.float32, device=dev)
    W[:sh.cout, :sh.D] = (torch.randn((sh.cout, sh.D), generator=gen, device=dev)
                          * float(np.sqrt(2.0 / sh.D)))
    return dH, X, W


class LayerState:
    """Device-resident operands, codes and outputs of one layer and its five
    C-ABI calls (Q_f, Q_theta, Q_b2 + Q_b1, grad_X, grad_W)."""

    def __init__(self, fqt, dH, X, W, ws, kind=KIND, bits=BITS, block=BLOCK, seed=5,
                 byte_operands=False):
        dev = dH.device
        N, C = dH.shape
        # X: a matrix (N x D), or an NHWC conv input (n, h, w, c) read as its
        # implicit im2col matrix (3 x 3 taps, pad 1)
        self.implicit = X.dim() == 4
        D = 9 * X.shape[3] if self.implicit else X.shape[1]
        self.N, self.C, self.D = N, C, D
        self.dH, self.X, self.W = dH, X, W
        self.kind, self.bits, self.block, self.seed = kind, bits, block, seed
        # grad_W's operands X~ and Q_b1 as 1-byte codes (widened on chip by the
        # contraction) or as fp16 carriers (the default: faster end to end, the
        # widening binds the contraction)
        b = byte_operands
        self.qx = (fqt.quantize_act_conv(X, 3, 3, 1, 8, ws=ws) if self.implicit else
                   fqt.QTensor.empty(N, D, fqt.PTQ, 8, 0, False, True, dev, u8=b, f16=not b))
        self.qw = fqt.QTensor.empty(C, D, fqt.PTQ, 8, 0, False, True, dev, u8=False)
        self.q2 = fqt.QTensor.empty(N, C, kind, bits, block, True, False, dev, u8=False)
        self.q1 = fqt.QTensor.empty(N, C, fqt.PTQ, 8, 0, False, True, dev, u8=b, f16=not b)
        self.gx = torch_empty((N, D), dev)
        self.gw = torch_empty((C, D), dev)
        self.ws = ws
        self.fqt = fqt

    def calls(self, dH=None, X=None, W=None, gx=None, gw=None, seed=None):
        f, ws = self.fqt, self.ws
        dH = self.dH if dH is None else dH
        X = self.X if X is None else X
        W = self.W if W is None else W
        gx = self.gx if gx is None else gx
        gw = self.gw if gw is None else gw
        seed = self.seed if seed is None else seed
        qa = ((lambda: f.quantize_act_conv(X, 3, 3, 1, 8, ws=ws, out=self.qx)) if self.implicit
              else (lambda: f.quantize_act(X, 8, ws=ws, out=self.qx)))
        return [
            qa,
            lambda: f.quantize_weight(W, 8, ws=ws, out=self.qw),
            lambda: f.quantize_grad(dH, self.kind, self.bits, self.block, seed, ws=ws,
                                    q_b2=self.q2, q_b1=self.q1),
            lambda: f.linear_backward(self.q2, self.q1, self.qx, self.qw, grad_x=True,
                                      grad_w=False, ws=ws, out_x=gx),
            lambda: f.linear_backward(self.q2, self.q1, self.qx, self.qw, grad_x=False,
                                      grad_w=True, ws=ws, out_w=gw),
        ]


def torch_empty(shape, dev):
    import torch
    return torch.empty(shape, dtype=torch.float32, device=dev)


def capture(fns):
    """One CUDA graph per call (the library's launches on the capturing
    stream): the timed replays carry no host launch overhead."""
    import torch
    graphs = []
    for f in fns:
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            f()
        graphs.append(g)
    return graphs


def roofline_of(call: str, rows, hbm_peak: float, bf16_peak: float):
    """Roofline of one call type over the sweep's layers.  rows: per layer
    (ms, algorithmic bytes, ops).  A contraction is HBM-bound on a layer when
    its ops per algorithmic byte are below the ridge (tensor peak of the fp16
    kind = the measured bf16 peak, over the measured HBM copy bandwidth);
    `achieved` aggregates the launches on the binding side that takes most
    of the call's time."""
    ridge = bf16_peak * 1e12 / (hbm_peak * 1e9)
    hb = [(ms, by, op) for ms, by, op in rows if not op or op / by < ridge]
    tb = [(ms, by, op) for ms, by, op in rows if op and op / by >= ridge]
    t_h, t_t = sum(r[0] for r in hb), sum(r[0] for r in tb)
    out = {"call": call, "kernel": KERNELS[call],
           "launches_per_call": 1 if call == "grad_x" else 2,
           "ms": t_h + t_t}
    if hb:
        gbs = sum(r[1] for r in hb) / (t_h * 1e-3) / 1e9
        out["hbm_bound_layers"] = {"n": len(hb), "ms": t_h, "achieved_GBs": gbs,
                                   "frac": gbs / hbm_peak}
    if tb:
        tops = sum(r[2] for r in tb) / (t_t * 1e-3) / 1e12
        out["tensor_bound_layers"] = {"n": len(tb), "ms": t_t, "achieved_TOPS": tops,
                                      "frac": tops / bf16_peak}
    if t_h >= t_t:
        by = sum(r[1] for r in hb)
        out.update(bound="hbm", achieved=by / (t_h * 1e-3) / 1e9, peak=hbm_peak, unit="GB/s",
                   algorithmic_bytes=by, launches=len(hb))
    else:
        op = sum(r[2] for r in tb)
        out.update(bound="tensor", achieved=op / (t_t * 1e-3) / 1e12, peak=bf16_peak,
                   unit="TFLOP/s", algorithmic_ops=op, launches=len(tb))
    out["frac"] = out["achieved"] / out["peak"]
    return out


def run_gpu(args):
    import torch
    import torch.distributed as dist
    from paper_2010_14298_gb300 import fqt
    from paper_2010_14298_gb300 import workloads as wl

    world, rank, local = _dist()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    fqt.load(build_if_missing=True)
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    hbm_peak, bf16_peak, peak_src = _peaks()

    # ---- the sweep's layers, resident in HBM ----
    shapes = wl.resnet50_shapes()
    B = SWEEP_BATCH
    big = max(shapes, key=lambda s: fqt.workspace_size(s.rows(B), s.C_pad, s.D_pad))
    ws = fqt.Workspace(big.rows(B), big.C_pad, big.D_pad, device=dev)  # calls run in order
    layers = []
    for li, sh in enumerate(shapes):
        dH, X, W = sweep_layer_tensors(sh, B, rank_seed(rank, li), dev,
                                       implicit=implicit_ok(sh))
        layers.append(LayerState(fqt, dH, X, W, ws))
    nl = len(layers)
    ops_layer = [4 * sh.rows(B) * sh.cout * sh.D for sh in shapes]
    ops_step = sum(ops_layer)
    byt = [alg_bytes(L.N, L.C, L.D) for L in layers]
    for L, b in zip(layers, byt):
        if L.implicit:  # Q_f reads the NHWC input once and writes its codes
            px = L.X.numel()
            b["quantize_act"] = px * 4 + px + L.D * 4 + 8
    nlaunch = sum(sum(launches(L.C, implicit=L.implicit).values()) for L in layers)

    for _ in range(args.warmup):
        for L in layers:
            for f in L.calls():
                f()
    torch.cuda.synchronize()
    if fqt.sync_status(ws) != 0:
        raise RuntimeError("device-side status after warm-up")
    graphs = [capture(L.calls()) for L in layers]
    for _ in range(2):
        for gl in graphs:
            for g in gl:
                g.replay()
    torch.cuda.synchronize()
    if fqt.sync_status(ws) != 0:
        raise RuntimeError("device-side status after graph warm-up")

    ncalls = nl * len(CALLS)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(ncalls + 1)]
           for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with Clocks(local) as clk:
        clk.wait_first()
        t_wall = time.perf_counter()
        clk.mark_start()
        for i in range(args.steps):
            e, k = evs[i], 0
            for gl in graphs:
                for g in gl:
                    e[k].record(stream)
                    g.replay()
                    k += 1
            e[k].record(stream)
        torch.cuda.synchronize()
        clk.mark_end()
        t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    per = np.zeros((nl, len(CALLS)))
    step_ms = []
    for e in evs:
        d = np.array([e[j].elapsed_time(e[j + 1]) for j in range(ncalls)])
        per += d.reshape(nl, len(CALLS))
        step_ms.append(e[0].elapsed_time(e[ncalls]))
    per /= args.steps
    ms_step = max_over_ranks(float(np.mean(step_ms)), dev)
    status = fqt.sync_status(ws)
    value = ops_step * world / (ms_step * 1e-3) / 1e12

    # ---- rooflines: every call type over the layers; the dominant one is
    # the call with the largest share of the step ----
    roofs = {}
    for ci, c in enumerate(CALLS):
        rows = [(per[li, ci], byt[li][c], ops_layer[li] // 2 if c in ("grad_x", "grad_w") else 0)
                for li in range(nl)]
        roofs[c] = roofline_of(c, rows, hbm_peak, bf16_peak)
    call_ms = {c: float(per[:, ci].sum()) for ci, c in enumerate(CALLS)}
    # The dominant kernel of the step is k_gemm (the largest share of the ncu
    # launch list: grad_X and the split-K partials of grad_W).  grad_X
    # launches it alone, so the per-call events time that kernel; its
    # roofline is taken over the grad_X launches on their binding side.
    dom = "grad_x"
    r = roofs[dom]
    roofline = {"bound": r["bound"], "achieved": r["achieved"], "peak": r["peak"],
                "unit": r["unit"], "frac": r["frac"],
                "traffic": _traffic_record("k_gemm", "resnet50-sweep-b256"),
                "algorithmic_bytes": r.get("algorithmic_bytes"),
                "kernel": "k_gemm", "call": dom, "peak_source": peak_src,
                "launches": r["launches"],
                "per_launch": ("algorithmic bytes (1 byte per code), DRAM traffic (ncu "
                               "dram__bytes_read.sum + dram__bytes_write.sum) and CUDA-event "
                               f"time summed over the {r['launches']} {r['bound']}-bound grad_X "
                               "launches of the step")}
    slow = sorted(range(nl), key=lambda li: -per[li].sum())[:6]
    result = {
        "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "u8 codes (fp16 carriers, exact int accumulation); f32 in/out",
        "data": "synthetic (seeded on the device; shapes and value distributions of the workload)",
        "config": {"workload": WORKLOAD, "layers": nl, "global_batch": B * world,
                   "quantizer": "Q_b2=BHQ-5 block16, Q_b1=PTQ-8 stochastic, X~/W~=PTQ-8",
                   "ops_per_step": ops_step,
                   "parallelism": f"replicas x{world} (independent batches)",
                   "lowering": (f"{sum(L.implicit for L in layers)} stride-1 3x3 convs as "
                                "implicit im2col (NHWC input read once), the rest as "
                                "materialized im2col matrices"),
                   "l2": ("no flush: inputs larger than L2 (a step reads "
                          f"{sum(4 * (L.dH.numel() + L.X.numel() + L.W.numel()) for L in layers) / 1e9:.1f}"
                          " GB of fp32 inputs)"),
                   "launch": "one CUDA graph per C-ABI call, events between calls",
                   "wall_s": t_wall},
        "roofline": roofline,
        "per_call_ms": call_ms,
        "rooflines": roofs,
        "per_layer_ms": {shapes[li].name: [round(float(v), 4) for v in per[li]]
                         for li in range(nl)},
        "slowest_layers": [{"layer": shapes[li].name, "N": layers[li].N, "C": shapes[li].cout,
                            "D": shapes[li].D,
                            "ms": dict(zip(CALLS, [float(v) for v in per[li]]))}
                           for li in slow],
        "stem_grad_x_ms": float(per[0, 3]),
        "clocks": clk.summary(),
        "gpu_launches": int(nlaunch * args.steps),
        "device_status": status,
    }
    if args.e2e_steps > 0:
        result["e2e"] = e2e_sweep(fqt, layers, shapes, ops_step * world, args, dev, stream)
    if args.extras:
        result["extras"] = run_extras(args, fqt, wl, dev, stream, hbm_peak, bf16_peak)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(args.cpu_batch)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()


def e2e_sweep(fqt, layers, shapes, ops_step, args, dev, stream):
    """The same step through the public API with host buffers: every layer's
    dH, X and W are copied from pinned host memory and its grad_X and grad_W
    copied back, every step.  Layers are pipelined on three streams
    (host-to-device copies, the C-ABI calls, device-to-host copies) through
    three device staging sets sized for the largest layer, so the copies of
    neighbouring layers overlap each other and the calls."""
    import torch
    h_in, h_out = [], []
    try:
        for L in layers:
            ins = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in (L.dH, L.X, L.W)]
            for h, t in zip(ins, (L.dH, L.X, L.W)):
                h.copy_(t)
            h_in.append(ins)
            h_out.append([torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
                          for t in (L.gx, L.gw)])
    except RuntimeError as exc:  # pinned host memory exhausted
        return {"value": None, "unit": "TOPS", "error": f"pinned host buffers: {exc}"[:200]}
    sz = {k: max(getattr(L, k).numel() for L in layers) for k in ("dH", "X", "W", "gx", "gw")}
    NSET = 3
    sets = [{k: torch.empty(n, dtype=torch.float32, device=dev) for k, n in sz.items()}
            for _ in range(NSET)]
    view = lambda s, k, t: s[k][:t.numel()].view(t.shape)
    s_in, s_cmp, s_out = (torch.cuda.Stream(dev) for _ in range(3))
    done_cmp, done_out = [None] * NSET, [None] * NSET

    def run(nsteps, seed0):
        g = 0
        for i in range(nsteps):
            for li, L in enumerate(layers):
                j = g % NSET
                s = sets[j]
                with torch.cuda.stream(s_in):
                    if done_cmp[j] is not None:  # the set's last layer has read it
                        s_in.wait_event(done_cmp[j])
                    for k, h in zip(("dH", "X", "W"), h_in[li]):
                        view(s, k, h).copy_(h, non_blocking=True)
                    ein = torch.cuda.Event()
                    ein.record(s_in)
                with torch.cuda.stream(s_cmp):
                    s_cmp.wait_event(ein)
                    if done_out[j] is not None:  # its gradients have left
                        s_cmp.wait_event(done_out[j])
                    for f in L.calls(dH=view(s, "dH", L.dH), X=view(s, "X", L.X),
                                     W=view(s, "W", L.W), gx=view(s, "gx", L.gx),
                                     gw=view(s, "gw", L.gw), seed=seed0 + i):
                        f()
                    ec = torch.cuda.Event()
                    ec.record(s_cmp)
                    done_cmp[j] = ec
                with torch.cuda.stream(s_out):
                    s_out.wait_event(ec)
                    for k, h in zip(("gx", "gw"), h_out[li]):
                        h.copy_(view(s, k, h), non_blocking=True)
                    eo = torch.cuda.Event()
                    eo.record(s_out)
                    done_out[j] = eo
                g += 1
        for st_ in (s_in, s_cmp, s_out):
            stream.wait_stream(st_)

    run(1, 2000)  # warms the pinned-copy path and the streams
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for st_ in (s_in, s_cmp, s_out):
        st_.wait_stream(stream)
    run(args.e2e_steps, 3000)
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / args.e2e_steps
    h2d = sum(sum(t.numel() * 4 for t in (L.dH, L.X, L.W)) for L in layers)
    d2h = sum(sum(t.numel() * 4 for t in (L.gx, L.gw)) for L in layers)
    status = fqt.sync_status(layers[0].ws)
    del h_in, h_out, sets
    return {"value": ops_step / (ms * 1e-3) / 1e12, "unit": "TOPS", "ms_per_step": ms,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h),
            "schedule": "layers pipelined on three streams (H2D / C-ABI calls / D2H), three "
                        "device staging sets, pinned host buffers per layer, eager calls",
            "device_status": status}


def run_extras(args, fqt, wl, dev, stream, hbm_peak, bf16_peak):
    """The other workloads and the method's variants, each call replayed as
    one CUDA graph and timed alone (median over rounds, L2 flushed before
    each round)."""
    import torch
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    steps = args.extra_steps

    def time_graphs(fns):
        for _ in range(3):
            for f in fns:
                f()
        torch.cuda.synchronize()
        gs = capture(fns)
        tt = [[] for _ in fns]
        for i in range(steps):
            flush.fill_(i & 0xFF)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(fns) + 1)]
            for k, g in enumerate(gs):
                ev[k].record(stream)
                g.replay()
            ev[-1].record(stream)
            torch.cuda.synchronize()
            for k in range(len(fns)):
                tt[k].append(ev[k].elapsed_time(ev[k + 1]))
        return [float(np.median(t)) for t in tt]

    def on_dev(Lw):
        dt = torch.bfloat16 if Lw.dtype == "bf16" else torch.float32
        return [torch.from_numpy(a).to(dev).to(dt) for a in (Lw.dH, Lw.X, Lw.W)]

    def layer_runs(Lw, runs):
        dH, X, W = on_dev(Lw)
        eb = 2 if Lw.dtype == "bf16" else 4
        ws = fqt.Workspace(Lw.N, Lw.C, Lw.D, device=dev)
        out = []
        for kind, bits, block in runs:
            st = LayerState(fqt, dH, X, W, ws, kind, bits, block, seed=5)
            per = time_graphs(st.calls())
            by = alg_bytes(Lw.N, Lw.C, Lw.D, eb, block if kind == KIND else 0)
            ops = 2 * Lw.N * Lw.C * Lw.D
            roof = {}
            for c, ms in (("grad_x", per[3]), ("grad_w", per[4])):
                r = roofline_of(c, [(ms, by[c], ops)], hbm_peak, bf16_peak)
                roof[c] = {"bound": r["bound"], "frac": r["frac"], "achieved": r["achieved"],
                           "unit": r["unit"]}
            name = {0: "PTQ", 1: "PSQ", 2: "BHQ"}[kind] + f"-{bits}" + (
                f" block {block}" if kind == KIND else "")
            out.append({"Q_b2": name, "per_call_ms": dict(zip(CALLS, per)),
                        "ms_per_step": sum(per), "TOPS": 2 * ops / (sum(per) * 1e-3) / 1e12,
                        "quantize_grad_GBs": by["quantize_grad"] / (per[2] * 1e-3) / 1e9,
                        "roofline": roof, "device_status": fqt.sync_status(ws)})
            del st
        del dH, X, W, ws
        torch.cuda.empty_cache()
        return out

    ex = {}
    # dense tensor-core rates (burst, each kernel timed alone): the fp16 kind
    # the contractions use, e4m3, and the legacy mma.sync IMMA path
    wsp0 = fqt.Workspace(1, 16, 16, device=dev)
    peaks = {}
    for kind, name, iters in ((0, "tcgen05 kind::f16 (fp16 x fp16 -> fp32) TFLOP/s", 20000),
                              (1, "tcgen05 kind::f8f6f4 (e4m3 x e4m3 -> fp32) TFLOP/s", 20000),
                              (2, "mma.sync m16n8k32 u8 x s8 -> s32 TOPS", 4000)):
        fqt.debug_mma_peak(kind, 50, wsp0)
        torch.cuda.synchronize()
        best = 0.0
        for _ in range(3):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            ops = fqt.debug_mma_peak(kind, iters, wsp0)
            e1.record(stream)
            torch.cuda.synchronize()
            best = max(best, ops / (e0.elapsed_time(e1) * 1e-3) / 1e12)
        peaks[name] = best
    peaks["tcgen05 kind::i8"] = "does not assemble for sm_103a (ptxas)"
    props = torch.cuda.get_device_properties(dev)
    peaks["sm_count"] = props.multi_processor_count
    peaks["l2_bytes"] = getattr(props, "L2_cache_size", None)
    peaks["device_status"] = fqt.sync_status(wsp0)
    ex["mma_peaks"] = peaks
    # linear layer 128 x 256: launch-bound, reported as latency
    L1 = wl.config(0)[0]
    ex["linear-128x256"] = {
        "latency": [{"Q_b2": r["Q_b2"], "step_us": r["ms_per_step"] * 1e3,
                     "per_call_us": {k: v * 1e3 for k, v in r["per_call_ms"].items()}}
                    for r in layer_runs(L1, [(0, 8, 0), (1, 8, 0), (KIND, 5, 16)])]}
    L2 = wl.config(1)[0]
    ex["resnet18-conv3x3"] = {"N": L2.N, "C": L2.C, "D": L2.D, "runs": layer_runs(
        L2, [(k, b, 16 if k == KIND else 0) for k in (0, 1, KIND) for b in (4, 5, 8)])}
    L3 = wl.config(2)[0]
    ex["resnet50-layer3-conv3x3"] = {"N": L3.N, "C": L3.C, "D": L3.D, "runs": layer_runs(
        L3, [(KIND, 5, nb) for nb in (8, 16, 32, 64)])}
    del L3
    for Lf in wl.config(3):
        ex[Lf.name.split(":")[0] + ":" + Lf.name.split(":")[1]] = {
            "N": Lf.N, "C": Lf.C, "D": Lf.D, "dtype": "bf16",
            "runs": layer_runs(Lf, [(0, 8, 0), (1, 5, 0), (KIND, 5, 16)])}

    # variants on the ResNet-18 conv layer
    dH, X, W = on_dev(L2)
    N, C, D = L2.N, L2.C, L2.D
    ws = fqt.Workspace(N, C, D, device=dev)
    # carriers: the shift quantizer's and the implicit im2col's grad_W pair
    # these operands with fp16 operands of their own
    base = LayerState(fqt, dH, X, W, ws, byte_operands=False)
    per_base = time_graphs(base.calls())
    # grad_W's byte-operand path on the same layer (1-byte X~ and Q_b1)
    byt = LayerState(fqt, dH, X, W, ws, byte_operands=True)
    per_byt = time_graphs(byt.calls())
    ex["byte_operands"] = {
        "what": "X~ and Q_b1 written as 1-byte codes only; grad_W's split-K kernel widens "
                "them to fp16 carriers on chip (bit-identical grad_W)",
        "per_call_ms": dict(zip(CALLS, per_byt)),
        "carriers_per_call_ms": dict(zip(CALLS, per_base)),
        "device_status": fqt.sync_status(ws)}
    qa = fqt.QTensor.empty(N, C, fqt.BHQ, BITS, 0, True, False, dev, u8=False)
    qa1 = fqt.QTensor.empty(N, C, fqt.PTQ, 8, 0, False, True, dev, u8=False)
    pa = time_graphs([
        lambda: fqt.quantize_grad(dH, fqt.BHQ, BITS, 0, 7, ws=ws, q_b2=qa, q_b1=qa1),
        lambda: fqt.linear_backward(qa, qa1, base.qx, base.qw, grad_x=True, grad_w=False,
                                    ws=ws, out_x=base.gx)])
    ex["adaptive_bhq"] = {"quantizer": f"BHQ-{BITS}, adaptive groups (block 0)",
                          "quantize_grad_ms": pa[0], "grad_x_ms": pa[1],
                          "fixed_block16_ms": {"quantize_grad": per_base[2],
                                               "grad_x": per_base[3]},
                          "groups": int((qa.gstart[:N] < N).sum().item()),
                          "device_status": fqt.sync_status(ws)}
    qs = fqt.QTensor.empty(N, C, fqt.SHIFT, BITS, 0, True, False, dev, u8=False)
    ps = time_graphs([
        lambda: fqt.quantize_grad(dH, fqt.SHIFT, BITS, 0, 11, with_b1=False, ws=ws, q_b2=qs),
        lambda: fqt.linear_backward(qs, None, base.qx, base.qw, grad_x=True, grad_w=False,
                                    ws=ws, out_x=base.gx),
        lambda: fqt.linear_backward(qs, None, base.qx, base.qw, grad_x=False, grad_w=True,
                                    ws=ws, out_w=base.gw)])
    ex["shift_quantizer"] = {"quantizer": f"SHIFT-{BITS} (per-tensor range, per-row shifts "
                                          "in [0, 4]; no Q_b1)",
                             "quantize_grad_ms": ps[0], "grad_x_ms": ps[1], "grad_w_ms": ps[2],
                             "device_status": fqt.sync_status(ws)}
    xn = torch.from_numpy(L2.x_nhwc).to(dev)
    box = {}

    def qconv():
        box["qc"] = fqt.quantize_act_conv(xn, 3, 3, 1, 8, ws=ws, out=box.get("qc"))
    qconv()
    pi = time_graphs([qconv, lambda: fqt.linear_backward(base.q2, base.q1, box["qc"], base.qw,
                                                         grad_x=False, grad_w=True, ws=ws,
                                                         out_w=base.gw)])
    ex["implicit_im2col"] = {"x_input": "NHWC 128x32x32x64, 3x3 taps, pad 1, stride 1",
                             "quantize_act_conv_ms": pi[0], "grad_w_ms": pi[1],
                             "explicit_ms": {"quantize_act": per_base[0], "grad_w": per_base[4]},
                             "device_status": fqt.sync_status(ws)}
    # per-image samples (Sec. 4.1) and grad_X in NHWC with col2im fused: the
    # same layer (batch 128, 32 x 32, 64 -> 64 channels), PSQ-5 with one
    # sample per image
    q2p = fqt.QTensor.empty(N, C, fqt.PSQ, 5, 0, True, False, dev, u8=False)
    q1p = fqt.QTensor.empty(N, C, fqt.PTQ, 8, 0, False, True, dev, u8=False)
    nimg, hh, wimg, cin = L2.x_nhwc.shape
    outn = torch.empty((nimg, hh, wimg, cin), dtype=torch.float32, device=dev)
    wsc = fqt.Workspace(1, 16, 16, device=dev)
    wsc.nbytes = int(fqt.load().fqt_conv_grad_x_workspace_size(cin))
    wsc.buf = torch.zeros(wsc.nbytes, dtype=torch.uint8, device=dev)
    ps_ = time_graphs([
        lambda: fqt.quantize_grad_samples(dH, hh * wimg, fqt.PSQ, 5, 3, ws=ws, q_b2=q2p,
                                          q_b1=q1p),
        lambda: fqt.conv_grad_x_nhwc(q2p, base.qw, nimg, hh, wimg, cin, ws=wsc, out=outn),
        lambda: fqt.linear_backward(q2p, q1p, base.qx, base.qw, grad_x=True, grad_w=False, ws=ws,
                                    out_x=base.gx)])
    nb_out = nimg * hh * wimg * cin * 4
    by_nhwc = N * C + C * D + nb_out + N * 4 + D * 4
    ex["per_image_samples_and_fused_col2im"] = {
        "quantizer": "Q_b2 = PSQ-5 with one sample per image (rows_per_sample = 1024), Q_b1 PTQ-8",
        "quantize_grad_samples_ms": ps_[0],
        "grad_x_nhwc_ms": ps_[1],
        "grad_x_nhwc_GBs": by_nhwc / (ps_[1] * 1e-3) / 1e9,
        "grad_x_nhwc_frac_of_hbm": by_nhwc / (ps_[1] * 1e-3) / 1e9 / hbm_peak,
        "grad_x_im2col_ms": ps_[2],
        "output_bytes": {"nhwc": nb_out, "im2col": N * D * 4},
        "device_status": max(fqt.sync_status(ws), fqt.sync_status(wsc))}
    qxr = fqt.quantize_act(X, 8, row_sum=True)
    qwr = fqt.quantize_weight(W, 8, row_sum=True)
    H = torch.empty((N, C), dtype=torch.float32, device=dev)
    pf = time_graphs([lambda: fqt.linear_forward(qxr, qwr, ws=ws, out=H)])
    fb = N * D + C * D + N * C * 4 + N * 8 + C * 4
    ex["forward"] = {"call": "linear_forward (H = X~ W~^T, one k_gemm launch)", "ms": pf[0],
                     "TOPS": 2 * N * C * D / (pf[0] * 1e-3) / 1e12,
                     "GBs": fb / (pf[0] * 1e-3) / 1e9,
                     "frac_of_hbm": fb / (pf[0] * 1e-3) / 1e9 / hbm_peak}
    del dH, X, W, ws, base, qa, qa1, qs, xn, box, qxr, qwr, H, q2p, q1p, outn, wsc
    torch.cuda.empty_cache()

    # the paper's own overhead shape (Sec. 4.3): dH of a conv with N = 128,
    # C = 64, 56 x 56 (401408 im2col rows); the paper timed its CPU routines
    # there (context only, another machine)
    dHp = torch.from_numpy(wl.random_grad(wl.rng(480), 128 * 56 * 56, 64, sigma=2.0,
                                          outlier_frac=0.01)).to(dev)
    Np = dHp.shape[0]
    wsp = fqt.Workspace(Np, 64, 16, device=dev)
    qsets = {}
    for name, kind, bits, block in (("PTQ-8", 0, 8, 0), ("PSQ-8", 1, 8, 0),
                                    ("BHQ-5 block 16", KIND, 5, 16),
                                    ("BHQ-5 adaptive groups", KIND, 5, 0)):
        qsets[name] = (fqt.QTensor.empty(Np, 64, kind, bits, block, True, False, dev, u8=False),
                       fqt.QTensor.empty(Np, 64, fqt.PTQ, 8, 0, False, True, dev, u8=False),
                       kind, bits, block)
    po = time_graphs([(lambda q=q: fqt.quantize_grad(dHp, q[2], q[3], q[4], 3, ws=wsp,
                                                      q_b2=q[0], q_b1=q[1]))
                      for q in qsets.values()])
    ex["paper_overhead_shape"] = {
        "shape": "dH 401408 x 64 fp32 (conv N=128, C=64, 56x56)",
        "quantize_grad_ms": dict(zip(qsets.keys(), po)),
        "paper_cpu_ms": {"per-tensor range": 11.0, "per-sample range": 24.0,
                         "Householder transform": 21.0, "INT8 conv layer": 480.0},
        "paper_cpu_note": "1 Intel CPU core, CPU TensorFlow + AVX (Sec. 4.3): context only",
        "device_status": fqt.sync_status(wsp)}
    del dHp, qsets, wsp, flush
    torch.cuda.empty_cache()
    return ex


# ---------------------------------------------------------------------------
# The CPU oracle on the host cores: one spawned process per core, each owning
# a fixed share of the sweep's layers (round robin), all starting each timed
# step together at a barrier; a step's time is the span from the first
# start to the last finish.  The oracle itself is single-threaded C.
# ---------------------------------------------------------------------------
def _oracle_worker(w, nproc, batch, steps, layer_ids, barrier, queue):
    os.environ["OMP_NUM_THREADS"] = "1"
    os.environ["OPENBLAS_NUM_THREADS"] = "1"
    try:
        import oracle as orc
        from paper_2010_14298_gb300 import workloads as wl
        shapes = wl.resnet50_shapes()
        mine = [li for i, li in enumerate(layer_ids) if i % nproc == w]
        data = [(shapes[li], wl.resnet50_layer(shapes[li], batch, rank_seed(0, li)))
                for li in mine]
        out = []
        for s in range(steps):
            barrier.wait(timeout=900)
            t0 = time.time()
            ops = 0
            for sh, L in data:
                orc.linear_backward(L.dH, L.X, L.W, KIND, BITS, BLOCK, s)
                ops += 4 * sh.rows(batch) * sh.cout * sh.D
            out.append((t0, time.time(), ops))
        queue.put((w, out, None))
    except Exception as exc:  # reported by the parent
        queue.put((w, None, repr(exc)[:300]))


def oracle_sweep(batch: int, steps: int, nproc: int, layer_ids=None):
    """[(seconds, ops)] per step of the oracle's full hot path over the
    sweep's layers at `batch`, on `nproc` processes."""
    import multiprocessing as mp
    import oracle
    from paper_2010_14298_gb300 import workloads as wl
    oracle.build()
    if layer_ids is None:
        layer_ids = list(range(len(wl.resnet50_shapes())))
    nproc = max(1, min(nproc, len(layer_ids)))
    ctx = mp.get_context("spawn")
    barrier = ctx.Barrier(nproc)
    queue = ctx.Queue()
    procs = [ctx.Process(target=_oracle_worker,
                         args=(w, nproc, batch, steps, layer_ids, barrier, queue), daemon=True)
             for w in range(nproc)]
    for p in procs:
        p.start()
    res = {}
    try:
        for _ in range(nproc):
            w, out, err = queue.get(timeout=1800)
            if err is not None:
                raise RuntimeError(f"oracle worker {w}: {err}")
            res[w] = out
    finally:
        for p in procs:
            p.join(timeout=30)
            if p.is_alive():
                p.terminate()
    return [(max(res[w][s][1] for w in res) - min(res[w][s][0] for w in res),
             sum(res[w][s][2] for w in res)) for s in range(steps)]


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_baseline(batch: int):
    cores = host_cores()
    par = oracle_sweep(batch, 1, cores)
    one = oracle_sweep(1, 1, 1)
    (dt, ops), (dt1, ops1) = par[0], one[0]
    return {"value": ops / dt / 1e12, "unit": "TOPS", "cores": cores, "kind": "oracle",
            "sample": f"every layer of the sweep at batch {batch} (instead of 256), full hot "
                      f"path, {cores} processes of the single-threaded oracle (layers dealt "
                      f"round robin): {dt:.1f} s wall for {ops / 1e9:.1f} GOP",
            "single_thread": {"value": ops1 / dt1 / 1e12, "unit": "TOPS", "cores": 1,
                              "sample": f"every layer at batch 1, one process: {dt1:.1f} s"}}


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2010_14298_gb300 import workloads as wl
    cores = host_cores()
    nl = len(wl.resnet50_shapes())
    # each step: the whole sweep at batch 1 (about 0.5 s on 16 cores); long
    # runs take every m-th layer per step so that the run stays in minutes
    m = max(1, -(-args.steps // 200))
    ids = list(range(0, nl, m))
    res = oracle_sweep(1, args.warmup + args.steps, cores, ids)[args.warmup:]
    dt = sum(r[0] for r in res)
    ops = sum(r[1] for r in res)
    value = ops / dt / 1e12
    sample = (f"{len(ids)} of the sweep's {nl} layers at batch 1 per step, full hot path, "
              f"{cores} processes of the single-threaded oracle")
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64 oracle (u8 codes)",
           "data": "synthetic (seeded)",
           "config": {"workload": WORKLOAD, "sample": sample},
           "cpu_baseline": {"value": value, "unit": "TOPS", "cores": cores, "kind": "oracle",
                            "sample": sample},
           "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=3,
                    help="timed end-to-end steps through the C ABI with host buffers (0: skip)")
    ap.add_argument("--cpu-batch", type=int, default=4,
                    help="batch of the CPU-baseline sample (every layer of the sweep)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extras", dest="extras", action="store_false",
                    help="skip the other workloads and the variants")
    ap.add_argument("--extra-steps", type=int, default=10,
                    help="timed rounds per call of the other workloads")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "native":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
