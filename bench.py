"""Benchmark of the FQT quantized backward on GB300.

One step = one pass of the whole hot path over one batch of the ResNet-18
3x3 conv backward (batch 128, 32x32, 64 -> 64 channels, im2col N = 131072,
C = 64, D = 576):
  X~ = Q_f(X), W~ = Q_theta(W)            (deterministic 8-bit PTQ)
  Q_b2(dH) = BHQ 5-bit, block 16; Q_b1(dH) = 8-bit stochastic PTQ
  grad_X = Q_b2(dH) W~,  grad_W = Q_b1(dH)^T X~
The reported value is quantized-backward throughput in TOPS: both
contractions count 2 N C D integer ops each.  Inputs are resident in HBM
when timing starts; L2 is flushed (256 MiB write) between timed steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

The reference arm times the CPU oracle on a bounded sample of the same
workload on the host cores.
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
WORKLOAD = "resnet18-conv3x3-b128-32x32-64ch (im2col N=131072, C=64, D=576)"
KIND, BITS, BLOCK = 2, 5, 16  # BHQ-5, block 16
CONFIG_INDEX = 1


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _traffic_record(kernel: str):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, if the
    summary was taken on the current kernel source."""
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
        if len(parts) >= 3 and parts[0] == kernel and parts[2] == digest:
            try:
                return float(parts[1])
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


def rank_seed(rank: int) -> int:
    """Seed of a rank's synthetic batch: replicas process independent batches
    of the same shapes and distributions (weak scaling)."""
    return 1234 + CONFIG_INDEX + 1000 * rank


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

    L = wl.config(CONFIG_INDEX, seed=rank_seed(rank))[0]
    N, C, D = L.N, L.C, L.D
    dH = torch.from_numpy(L.dH).to(dev)
    X = torch.from_numpy(L.X).to(dev)
    W = torch.from_numpy(L.W).to(dev)
    ws = fqt.Workspace(N, C, D, device=dev)
    ws_fx = fqt.Workspace(N, D, 16, device=dev)
    ws_fw = fqt.Workspace(C, D, 16, device=dev)
    # the backward consumes the fp16 carriers of the codes (2 bytes per code)
    qx = fqt.QTensor.empty(N, D, fqt.PTQ, 8, 0, False, True, dev, u8=False)
    qw = fqt.QTensor.empty(C, D, fqt.PTQ, 8, 0, False, True, dev, u8=False)
    q2 = fqt.QTensor.empty(N, C, KIND, BITS, BLOCK, True, False, dev, u8=False)
    q1 = fqt.QTensor.empty(N, C, fqt.PTQ, 8, 0, False, True, dev, u8=False)
    gx = torch.empty((N, D), dtype=torch.float32, device=dev)
    gw = torch.empty((C, D), dtype=torch.float32, device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)
    names = ["quantize_act", "quantize_weight", "quantize_grad", "grad_x", "grad_w"]
    # forward PTQ of X and of W: range + codes; Q_b2 / Q_b1: range +
    # warp-per-block BHQ quantizer; grad_X: one contraction; grad_W:
    # contraction + split-K reduction
    launches_per_call = [2, 2, 2, 1, 2]

    def calls(seed):
        return [
            lambda: fqt.quantize_act(X, 8, ws=ws_fx, out=qx),
            lambda: fqt.quantize_weight(W, 8, ws=ws_fw, out=qw),
            lambda: fqt.quantize_grad(dH, KIND, BITS, BLOCK, seed, ws=ws, q_b2=q2, q_b1=q1),
            lambda: fqt.linear_backward(q2, q1, qx, qw, grad_x=True, grad_w=False, ws=ws,
                                        out_x=gx),
            lambda: fqt.linear_backward(q2, q1, qx, qw, grad_x=False, grad_w=True, ws=ws,
                                        out_w=gw),
        ]

    graphs = None

    def step(seed, evs=None):
        def mark(i):
            if evs is not None:
                evs[i].record(stream)
        fns = [g.replay for g in graphs] if graphs is not None else calls(seed)
        for i, f in enumerate(fns):
            mark(i)
            f()
        mark(5)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    if fqt.sync_status(ws) != 0:
        raise RuntimeError("device-side status after warm-up")
    if not args.eager:
        # one CUDA graph per call (the library's launches on the capturing
        # stream), so the timed steps carry no host launch overhead; the
        # gradient quantizer's seed is fixed at capture
        graphs = []
        for f in calls(1000):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            graphs.append(g)
        for i in range(2):
            step(0)
        torch.cuda.synchronize()
        if fqt.sync_status(ws) != 0:
            raise RuntimeError("device-side status after graph warm-up")
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(6)]
           for _ in range(args.steps)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize()
    with Clocks(local) as clk:
        clk.wait_first()
        t_wall = time.perf_counter()
        clk.mark_start()
        for i in range(args.steps):
            flush.fill_(i & 0xFF)  # evict L2 between timed steps
            step(1000 + i, evs[i])
        torch.cuda.synchronize()
        clk.mark_end()
        t_wall = time.perf_counter() - t_wall
    if world > 1:
        dist.barrier()
    per_call = np.zeros(5)
    step_ms = []
    for e in evs:
        d = [e[j].elapsed_time(e[j + 1]) for j in range(5)]
        per_call += np.array(d)
        step_ms.append(sum(d))
    ms_step = float(np.mean(step_ms))
    per_call /= args.steps
    ms_step = max_over_ranks(ms_step, dev)
    status = fqt.sync_status(ws)

    ops_step = 2 * 2 * N * C * D  # both contractions
    value = ops_step * world / (ms_step * 1e-3) / 1e12

    # ---- roofline of the dominant kernel (largest share of the step) ----
    hbm_peak, peak_src = _peaks()
    # algorithmic bytes: each input read once, each output written once;
    # codes travel as 2-byte fp16 carriers
    cb = 2
    alg_bytes = {
        "quantize_act": N * D * 4 + N * D * cb + D * 4,
        "quantize_weight": C * D * 4 + C * D * cb + D * 4,
        "quantize_grad": N * C * 4 + 2 * N * C * cb + N * (4 + 4 + 4 + 8) + (N // BLOCK) * 4 + C * 4,
        "grad_x": N * C * cb + C * D * cb + N * D * 4 + N * 12 + (N // BLOCK) * 4 + D * 4,
        "grad_w": N * C * cb + N * D * cb + C * D * 4 + (C + D) * 4,
    }
    kern_of = {"quantize_act": "k_range + k_fwd_codes", "quantize_weight": "k_range + k_fwd_codes",
               "quantize_grad": "k_range + k_bhq_warp", "grad_x": "k_gemm",
               "grad_w": "k_gradw + k_reduce"}
    # The dominant kernel is the grad_X contraction (k_gemm, the largest
    # share of the ncu launch list); it is the only kernel of its call, so
    # the call's events time it alone.  The other calls launch two kernels
    # each; their whole-call bandwidth is reported beside it.
    dom = "grad_x"
    achieved = alg_bytes[dom] / (per_call[names.index(dom)] * 1e-3) / 1e9
    traffic = _traffic_record(dom)
    quant_gbs = alg_bytes["quantize_grad"] / (per_call[2] * 1e-3) / 1e9
    call_gbs = {k: alg_bytes[k] / (per_call[i] * 1e-3) / 1e9 for i, k in enumerate(names)}

    # ---- end to end through the public API with host buffers ----
    # Every step copies its inputs (dH, X, W) from pinned host memory, runs
    # the five C-ABI calls and copies both gradients back.  Steps are
    # pipelined two deep on three streams (host-to-device copies, calls,
    # device-to-host copies) with double-buffered device inputs and outputs,
    # so the copies of neighbouring steps overlap each other and the calls.
    e2e = None
    if args.e2e_steps > 0:
        h_dH = torch.from_numpy(L.dH).pin_memory()
        h_X = torch.from_numpy(L.X).pin_memory()
        h_W = torch.from_numpy(L.W).pin_memory()
        h_gx = torch.empty((N, D), dtype=torch.float32).pin_memory()
        h_gw = torch.empty((C, D), dtype=torch.float32).pin_memory()
        sets = [dict(dH=dH, X=X, W=W, gx=gx, gw=gw),
                dict(dH=torch.empty_like(dH), X=torch.empty_like(X), W=torch.empty_like(W),
                     gx=torch.empty_like(gx), gw=torch.empty_like(gw))]
        s_cmp = torch.cuda.Stream(dev)
        # each direction's copies can be split by rows over several streams
        # (several copy engines); one stream per direction measured fastest
        ncs = max(1, args.e2e_copy_streams)
        s_ins = [torch.cuda.Stream(dev) for _ in range(ncs)]
        s_outs = [torch.cuda.Stream(dev) for _ in range(ncs)]

        def split_rows(t):
            n_ = t.shape[0]
            step_ = (n_ + ncs - 1) // ncs
            return [t[i:i + step_] for i in range(0, n_, step_)]

        def e2e_calls(b, seed):
            return [lambda: fqt.quantize_act(b["X"], 8, ws=ws_fx, out=qx),
                    lambda: fqt.quantize_weight(b["W"], 8, ws=ws_fw, out=qw),
                    lambda: fqt.quantize_grad(b["dH"], KIND, BITS, BLOCK, seed, ws=ws, q_b2=q2,
                                              q_b1=q1),
                    lambda: fqt.linear_backward(q2, q1, qx, qw, ws=ws, out_x=b["gx"],
                                                out_w=b["gw"])]

        def run_e2e(nsteps, seed0):
            done_cmp, done_out = [None, None], [None, None]
            for i in range(nsteps):
                b = sets[i & 1]
                eins = []
                for si, s_in in enumerate(s_ins):
                    with torch.cuda.stream(s_in):
                        if done_cmp[i & 1] is not None:  # step i-2 has read these inputs
                            s_in.wait_event(done_cmp[i & 1])
                        for k, hsrc in (("dH", h_dH), ("X", h_X), ("W", h_W)):
                            dst_, src_ = split_rows(b[k]), split_rows(hsrc)
                            if si < len(dst_):
                                dst_[si].copy_(src_[si], non_blocking=True)
                        ein = torch.cuda.Event()
                        ein.record(s_in)
                        eins.append(ein)
                with torch.cuda.stream(s_cmp):
                    for ein in eins:
                        s_cmp.wait_event(ein)
                    if done_out[i & 1] is not None:  # step i-2's gradients have left
                        for eo in done_out[i & 1]:
                            s_cmp.wait_event(eo)
                    for f in e2e_calls(b, seed0 + i):
                        f()
                    ec = torch.cuda.Event()
                    ec.record(s_cmp)
                    done_cmp[i & 1] = ec
                eos = []
                for si, s_out in enumerate(s_outs):
                    with torch.cuda.stream(s_out):
                        s_out.wait_event(ec)
                        for hdst, k in ((h_gx, "gx"), (h_gw, "gw")):
                            dst_, src_ = split_rows(hdst), split_rows(b[k])
                            if si < len(dst_):
                                dst_[si].copy_(src_[si], non_blocking=True)
                        eo = torch.cuda.Event()
                        eo.record(s_out)
                        eos.append(eo)
                done_out[i & 1] = eos
            for st_ in s_ins + [s_cmp] + s_outs:
                stream.wait_stream(st_)

        run_e2e(2, 2000)  # warms the pinned-copy path and the streams
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        flush.fill_(7)
        torch.cuda.synchronize()
        e0.record(stream)
        for st_ in s_ins + [s_cmp] + s_outs:
            st_.wait_stream(stream)
        run_e2e(args.e2e_steps, 3000)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1) / args.e2e_steps
        e2e = {"value": ops_step * world / (e2e_ms * 1e-3) / 1e12, "unit": "TOPS",
               "ms_per_step": e2e_ms,
               "h2d_bytes_per_step": int((N * C + N * D + C * D) * 4),
               "d2h_bytes_per_step": int((N * D + C * D) * 4),
               "schedule": ("2-deep pipeline: H2D / C-ABI calls / D2H on three streams, "
                            "double-buffered device inputs and outputs, eager calls" if ncs == 1 else
                            f"2-deep pipeline: H2D on {ncs} streams / C-ABI calls / D2H on {ncs} "
                            "streams (each copy split by rows), double-buffered device inputs and "
                            "outputs, eager calls")}

    # ---- the quantized forward GEMM H = X~ W~^T on the same layer (the
    # contraction core with the roles renamed), timed alone ----
    fwd = None
    if args.forward_steps > 0:
        qxr = fqt.quantize_act(X, 8, row_sum=True)
        qwr = fqt.quantize_weight(W, 8, row_sum=True)
        H = torch.empty((N, C), dtype=torch.float32, device=dev)
        wsf = fqt.Workspace(1, 16, 16, device=dev)
        for _ in range(3):
            fqt.linear_forward(qxr, qwr, ws=wsf, out=H)
        tf = []
        for i in range(args.forward_steps):
            flush.fill_(i & 0xFF)
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            fqt.linear_forward(qxr, qwr, ws=wsf, out=H)
            e1.record(stream)
            torch.cuda.synchronize()
            tf.append(e0.elapsed_time(e1))
        fwd_ms = float(np.median(tf))
        fwd_bytes = N * D * cb + C * D * cb + N * C * 4 + N * 8 + C * 4
        fwd = {"call": "linear_forward (H = X~ W~^T, one k_gemm launch)", "ms": fwd_ms,
               "TOPS": 2 * N * C * D / (fwd_ms * 1e-3) / 1e12,
               "algorithmic_bytes": fwd_bytes,
               "GBs": fwd_bytes / (fwd_ms * 1e-3) / 1e9,
               "frac_of_hbm": fwd_bytes / (fwd_ms * 1e-3) / 1e9 / hbm_peak,
               "device_status": fqt.sync_status(wsf)}

    # ---- adaptive BHQ groups (App. D.5) on the same layer: Q_b2 with the
    # grouping chosen for this batch (sort, estimate, layout, group
    # quantizer), then grad_X (contraction + the groups' reflection pass);
    # one CUDA graph per call, timed alone ----
    ada = None
    if args.adaptive_steps > 0:
        qa = fqt.QTensor.empty(N, C, fqt.BHQ, BITS, 0, True, False, dev, u8=False)
        qa1 = fqt.QTensor.empty(N, C, fqt.PTQ, 8, 0, False, True, dev, u8=False)
        fa = [lambda: fqt.quantize_grad(dH, fqt.BHQ, BITS, 0, 7, ws=ws, q_b2=qa, q_b1=qa1),
              lambda: fqt.linear_backward(qa, qa1, qx, qw, grad_x=True, grad_w=False, ws=ws,
                                          out_x=gx)]
        for _ in range(3):
            for f in fa:
                f()
        torch.cuda.synchronize()
        ga = []
        for f in fa:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            ga.append(g)
        ta = [[], []]
        for i in range(args.adaptive_steps):
            flush.fill_(i & 0xFF)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
            ev[0].record(stream)
            ga[0].replay()
            ev[1].record(stream)
            ga[1].replay()
            ev[2].record(stream)
            torch.cuda.synchronize()
            ta[0].append(ev[0].elapsed_time(ev[1]))
            ta[1].append(ev[1].elapsed_time(ev[2]))
        G = int((qa.gstart[:N] < N).sum().item())
        grouped = int((qa.gsize > 1).sum().item())
        ada = {"quantizer": f"BHQ-{BITS}, adaptive groups (block 0)",
               "quantize_grad_ms": float(np.median(ta[0])),
               "grad_x_ms": float(np.median(ta[1])),
               "fixed_block16_ms": {"quantize_grad": float(per_call[2]),
                                    "grad_x": float(per_call[3])},
               "groups": G, "rows_in_multirow_groups": grouped,
               "launches": {"quantize_grad": 10, "grad_x": 3},
               "device_status": fqt.sync_status(ws)}

    # ---- the per-sample power-of-two shift quantizer (Sec. 4.3) on the same
    # layer: one code set feeds both contractions (no Q_b1); one CUDA graph
    # per call, timed alone ----
    shf = None
    if args.shift_steps > 0:
        qs = fqt.QTensor.empty(N, C, fqt.SHIFT, BITS, 0, True, False, dev, u8=False)
        fs = [lambda: fqt.quantize_grad(dH, fqt.SHIFT, BITS, 0, 11, with_b1=False, ws=ws,
                                        q_b2=qs),
              lambda: fqt.linear_backward(qs, None, qx, qw, grad_x=True, grad_w=False, ws=ws,
                                          out_x=gx),
              lambda: fqt.linear_backward(qs, None, qx, qw, grad_x=False, grad_w=True, ws=ws,
                                          out_w=gw)]
        for _ in range(3):
            for f in fs:
                f()
        torch.cuda.synchronize()
        gs_ = []
        for f in fs:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            gs_.append(g)
        tsh = [[], [], []]
        for i in range(args.shift_steps):
            flush.fill_(i & 0xFF)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            for k in range(3):
                ev[k].record(stream)
                gs_[k].replay()
            ev[3].record(stream)
            torch.cuda.synchronize()
            for k in range(3):
                tsh[k].append(ev[k].elapsed_time(ev[k + 1]))
        sh = qs.shift.cpu().numpy()
        shf = {"quantizer": f"SHIFT-{BITS} (per-tensor range, per-row shifts in [0, 4])",
               "quantize_grad_ms": float(np.median(tsh[0])),
               "grad_x_ms": float(np.median(tsh[1])),
               "grad_w_ms": float(np.median(tsh[2])),
               "bifurcated_bhq16_ms": {"quantize_grad": float(per_call[2]),
                                       "grad_x": float(per_call[3]),
                                       "grad_w": float(per_call[4])},
               "rows_per_shift": [int((sh == k).sum()) for k in range(5)],
               "launches": {"quantize_grad": 2, "grad_x": 1, "grad_w": 2},
               "device_status": fqt.sync_status(ws)}

    # ---- the same step with X~ as an implicit im2col operand: the forward
    # PTQ reads the NHWC input once (the im2col matrix is never formed) and
    # grad_W reads its boxes at shifted pixel coordinates; codes and grad_W
    # are bit-identical to the explicit path ----
    imp = None
    if args.implicit_steps > 0 and L.x_nhwc is not None:
        xn = torch.from_numpy(L.x_nhwc).to(dev)
        nb, hh, ww, cc = L.x_nhwc.shape
        qc = None

        def qconv():
            nonlocal qc
            qc = fqt.quantize_act_conv(xn, 3, 3, 1, 8, ws=ws_fx, out=qc)
        qconv()
        fi = [qconv,
              lambda: fqt.quantize_weight(W, 8, ws=ws_fw, out=qw),
              lambda: fqt.quantize_grad(dH, KIND, BITS, BLOCK, 1000, ws=ws, q_b2=q2, q_b1=q1),
              lambda: fqt.linear_backward(q2, q1, qx, qw, grad_x=True, grad_w=False, ws=ws,
                                          out_x=gx),
              lambda: fqt.linear_backward(q2, q1, qc, qw, grad_x=False, grad_w=True, ws=ws,
                                          out_w=gw)]
        for _ in range(3):
            for f in fi:
                f()
        torch.cuda.synchronize()
        gi = []
        for f in fi:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            gi.append(g)
        ti = [[] for _ in fi]
        for i in range(args.implicit_steps):
            flush.fill_(i & 0xFF)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(fi) + 1)]
            for k in range(len(fi)):
                ev[k].record(stream)
                gi[k].replay()
            ev[-1].record(stream)
            torch.cuda.synchronize()
            for k in range(len(fi)):
                ti[k].append(ev[k].elapsed_time(ev[k + 1]))
        per = [float(np.median(t)) for t in ti]
        ms_imp = sum(per)
        imp = {"x_input": f"NHWC {nb}x{hh}x{ww}x{cc}, 3x3 taps, pad 1, stride 1",
               "per_call_ms": dict(zip(["quantize_act_conv", "quantize_weight", "quantize_grad",
                                        "grad_x", "grad_w"], per)),
               "ms_per_step": ms_imp,
               "TOPS": ops_step / (ms_imp * 1e-3) / 1e12,
               "explicit_ms": {"quantize_act": float(per_call[0]), "grad_w": float(per_call[4])},
               "launches_per_step": 10,
               "device_status": fqt.sync_status(ws)}

    def time_graphs(fns, steps):
        """Median ms of each call, replayed as one CUDA graph per call, L2
        flushed before each round."""
        for _ in range(3):
            for f in fns:
                f()
        torch.cuda.synchronize()
        gs_ = []
        for f in fns:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g):
                f()
            gs_.append(g)
        tt = [[] for _ in fns]
        for i in range(steps):
            flush.fill_(i & 0xFF)
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(len(fns) + 1)]
            for k, g in enumerate(gs_):
                ev[k].record(stream)
                g.replay()
            ev[-1].record(stream)
            torch.cuda.synchronize()
            for k in range(len(fns)):
                tt[k].append(ev[k].elapsed_time(ev[k + 1]))
        return [float(np.median(t)) for t in tt]

    bf16_peak = 1862.7
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            bf16_peak = float(json.load(f)["bf16_tflops"])
    except Exception:
        pass

    # ---- the other full-size workloads: one backward step per layer, each
    # contraction against its binding roofline (HBM bytes with 2-byte code
    # carriers, or the tensor peak of the fp16 kind = the measured bf16 peak) ----
    others = None
    if args.config_steps > 0:
        others = []
        for cfg in (2, 3):
            for Lo in wl.config(cfg):
                No, Co, Do = Lo.N, Lo.C, Lo.D
                dt = torch.bfloat16 if Lo.dtype == "bf16" else torch.float32
                to = lambda a: torch.from_numpy(a).to(dev).to(dt)
                dHo, Xo, Wo = to(Lo.dH), to(Lo.X), to(Lo.W)
                wso = fqt.Workspace(No, Co, Do, device=dev)
                qxo = fqt.QTensor.empty(No, Do, fqt.PTQ, 8, 0, False, True, dev, u8=False)
                qwo = fqt.QTensor.empty(Co, Do, fqt.PTQ, 8, 0, False, True, dev, u8=False)
                q2o = fqt.QTensor.empty(No, Co, fqt.BHQ, 5, 16, True, False, dev, u8=False)
                q1o = fqt.QTensor.empty(No, Co, fqt.PTQ, 8, 0, False, True, dev, u8=False)
                gxo = torch.empty((No, Do), dtype=torch.float32, device=dev)
                gwo = torch.empty((Co, Do), dtype=torch.float32, device=dev)
                wfx = fqt.Workspace(No, Do, 16, device=dev)
                wfw = fqt.Workspace(Co, Do, 16, device=dev)
                fo = [lambda: fqt.quantize_act(Xo, 8, ws=wfx, out=qxo),
                      lambda: fqt.quantize_weight(Wo, 8, ws=wfw, out=qwo),
                      lambda: fqt.quantize_grad(dHo, fqt.BHQ, 5, 16, 5, ws=wso, q_b2=q2o,
                                                q_b1=q1o),
                      lambda: fqt.linear_backward(q2o, q1o, qxo, qwo, grad_x=True, grad_w=False,
                                                  ws=wso, out_x=gxo),
                      lambda: fqt.linear_backward(q2o, q1o, qxo, qwo, grad_x=False, grad_w=True,
                                                  ws=wso, out_w=gwo)]
                per = time_graphs(fo, args.config_steps)
                ops = 2 * No * Co * Do
                eb = 2 if Lo.dtype == "bf16" else 4
                bytes_x = No * Co * 2 + Co * Do * 2 + No * Do * 4 + No * 12 + (No // 16) * 4
                bytes_w = No * Co * 2 + No * Do * 2 + Co * Do * 4 + (Co + Do) * 4
                roof = {}
                for name, ms, by in (("grad_x", per[3], bytes_x), ("grad_w", per[4], bytes_w)):
                    gbs = by / (ms * 1e-3) / 1e9
                    tops = ops / (ms * 1e-3) / 1e12
                    hbm_bound = ops / by < bf16_peak * 1e12 / (hbm_peak * 1e9)
                    roof[name] = {"bound": "hbm" if hbm_bound else "tensor", "ms": ms,
                                  "TOPS": tops, "GBs": gbs,
                                  "frac": gbs / hbm_peak if hbm_bound else tops / bf16_peak,
                                  "ops_per_byte": ops / by}
                others.append({"workload": Lo.name, "N": No, "C": Co, "D": Do,
                               "dtype": Lo.dtype, "quantizer": "BHQ-5 block 16 + Q_b1 PTQ-8",
                               "per_call_ms": dict(zip(["quantize_act", "quantize_weight",
                                                        "quantize_grad", "grad_x", "grad_w"],
                                                       per)),
                               "ms_per_step": sum(per),
                               "TOPS": 2 * ops / (sum(per) * 1e-3) / 1e12,
                               "quantize_grad_GBs": (No * Co * eb + 2 * No * Co * 2 + No * 20)
                               / (per[2] * 1e-3) / 1e9,
                               "roofline": roof, "device_status": fqt.sync_status(wso)})
                del dHo, Xo, Wo, qxo, qwo, q2o, q1o, gxo, gwo, wso, wfx, wfw
                torch.cuda.empty_cache()

    # ---- the full ResNet-50 backward sweep at batch 256, 224 x 224: every conv
    # (and the fc) lowered to im2col, BHQ-5/16 + Q_b1 PTQ-8 gradients, 8-bit
    # X~ and W~; inputs drawn on the device from the same recipe as
    # workloads.resnet50_layer (the host draw is 40+ GB) ----
    sweep = None
    if args.sweep_steps > 0:
        import torch.nn.functional as F
        layers_out = []
        tot = {"quantize_act": 0.0, "quantize_weight": 0.0, "quantize_grad": 0.0,
               "grad_x": 0.0, "grad_w": 0.0}
        ops_all = 0
        st_all = 0
        bsz = 256
        for li, sh in enumerate(wl.resnet50_shapes()):
            gen = torch.Generator(device=dev)
            gen.manual_seed(1234 + 4 + li)
            Ns, Dp, Cp = sh.rows(bsz), sh.D_pad, sh.C_pad
            x = torch.rand((bsz, sh.cin, sh.h, sh.h), generator=gen, device=dev) * 2.0 - 1.0
            cols = F.unfold(x, sh.k, padding=sh.pad, stride=sh.stride)
            del x
            Xs = torch.zeros((Ns, Dp), dtype=torch.float32, device=dev)
            Xs[:, :sh.D] = cols.view(bsz, sh.cin, sh.k * sh.k, -1).permute(0, 3, 2, 1).reshape(Ns, sh.D)
            del cols
            dHs = torch.zeros((Ns, Cp), dtype=torch.float32, device=dev)
            dHs[:, :sh.cout] = (torch.randn((Ns, sh.cout), generator=gen, device=dev)
                                * torch.exp(2.0 * torch.randn((Ns, 1), generator=gen, device=dev)))
            Ws = torch.zeros((Cp, Dp), dtype=torch.float32, device=dev)
            Ws[:sh.cout, :sh.D] = (torch.randn((sh.cout, sh.D), generator=gen, device=dev)
                                   * float(np.sqrt(2.0 / sh.D)))
            wss = fqt.Workspace(Ns, Cp, Dp, device=dev)
            qxs = fqt.QTensor.empty(Ns, Dp, fqt.PTQ, 8, 0, False, True, dev, u8=False)
            qws = fqt.QTensor.empty(Cp, Dp, fqt.PTQ, 8, 0, False, True, dev, u8=False)
            q2s = fqt.QTensor.empty(Ns, Cp, fqt.BHQ, 5, 16, True, False, dev, u8=False)
            q1s = fqt.QTensor.empty(Ns, Cp, fqt.PTQ, 8, 0, False, True, dev, u8=False)
            gxs = torch.empty((Ns, Dp), dtype=torch.float32, device=dev)
            gws = torch.empty((Cp, Dp), dtype=torch.float32, device=dev)
            wfxs = fqt.Workspace(Ns, Dp, 16, device=dev)
            wfws = fqt.Workspace(Cp, Dp, 16, device=dev)
            fs = [lambda: fqt.quantize_act(Xs, 8, ws=wfxs, out=qxs),
                  lambda: fqt.quantize_weight(Ws, 8, ws=wfws, out=qws),
                  lambda: fqt.quantize_grad(dHs, fqt.BHQ, 5, 16, 5, ws=wss, q_b2=q2s, q_b1=q1s),
                  lambda: fqt.linear_backward(q2s, q1s, qxs, qws, grad_x=True, grad_w=False,
                                              ws=wss, out_x=gxs),
                  lambda: fqt.linear_backward(q2s, q1s, qxs, qws, grad_x=False, grad_w=True,
                                              ws=wss, out_w=gws)]
            per = time_graphs(fs, args.sweep_steps)
            for k_, v_ in zip(tot, per):
                tot[k_] += v_
            ops_l = 2 * 2 * Ns * sh.cout * sh.D
            ops_all += ops_l
            st_all |= fqt.sync_status(wss)
            layers_out.append({"layer": sh.name, "N": Ns, "C": sh.cout, "D": sh.D,
                               "backward_ms": per[2] + per[3] + per[4], "grad_x_ms": per[3],
                               "TOPS": ops_l / ((per[3] + per[4]) * 1e-3) / 1e12})
            del Xs, dHs, Ws, wss, qxs, qws, q2s, q1s, gxs, gws, wfxs, wfws
            torch.cuda.empty_cache()
        bwd = tot["quantize_grad"] + tot["grad_x"] + tot["grad_w"]
        slow = sorted(layers_out, key=lambda r: -r["backward_ms"])[:5]
        sweep = {"workload": "ResNet-50 v1.5 backward sweep, batch 256, 224 x 224: 53 convs + fc "
                             "via im2col (stem D 147 -> 160 and fc C 1000 -> 1008 zero-padded)",
                 "layers": len(layers_out), "quantizer": "BHQ-5 block 16 + Q_b1 PTQ-8; X~, W~ PTQ-8",
                 "backward_ms": bwd, "ops": ops_all, "TOPS": ops_all / (bwd * 1e-3) / 1e12,
                 "per_call_ms_sum": tot,
                 "forward_quantizers_ms": tot["quantize_act"] + tot["quantize_weight"],
                 # the stem's grad_X (w.r.t. the image) is not needed in training
                 "stem_grad_x_ms": next(r for r in layers_out if r["layer"] == "conv1")["grad_x_ms"],
                 "slowest_layers": slow, "device_status": st_all}

    # ---- the paper's own overhead shape (Sec. 4.3): a conv layer with
    # N = 128, C = 64, 56 x 56, i.e. dH of 401408 im2col rows x 64; the paper
    # timed its CPU routines there (context only, another machine) ----
    ovh = None
    if args.config_steps > 0:
        gp = wl.rng(480)
        dHp = torch.from_numpy(wl.random_grad(gp, 128 * 56 * 56, 64, sigma=2.0,
                                              outlier_frac=0.01)).to(dev)
        Np = dHp.shape[0]
        wsp = fqt.Workspace(Np, 64, 16, device=dev)
        qsets = {}
        for name, kind, bits, block in (("PTQ-8", fqt.PTQ, 8, 0), ("PSQ-8", fqt.PSQ, 8, 0),
                                        ("BHQ-5 block 16", fqt.BHQ, 5, 16),
                                        ("BHQ-5 adaptive groups", fqt.BHQ, 5, 0)):
            qsets[name] = (fqt.QTensor.empty(Np, 64, kind, bits, block, True, False, dev, u8=False),
                           fqt.QTensor.empty(Np, 64, fqt.PTQ, 8, 0, False, True, dev, u8=False),
                           kind, bits, block)
        fns = [(lambda q=q: fqt.quantize_grad(dHp, q[2], q[3], q[4], 3, ws=wsp, q_b2=q[0],
                                              q_b1=q[1])) for q in qsets.values()]
        per = time_graphs(fns, args.config_steps)
        ovh = {"shape": "dH 401408 x 64 fp32 (conv N=128, C=64, 56x56)",
               "quantize_grad_ms": dict(zip(qsets.keys(), per)),
               "includes": "range pass, scales / transform, SR of Q_b2 and of the 8-bit Q_b1, "
                           "packing, row and column sums (and the grouping, adaptive)",
               "paper_cpu_ms": {"per-tensor range": 11.0, "per-sample range": 24.0,
                                "Householder transform": 21.0, "BHQ construction": 0.003,
                                "INT8 conv layer": 480.0},
               "paper_cpu_note": "1 Intel CPU core, CPU TensorFlow + AVX (Sec. 4.3): context only",
               "device_status": fqt.sync_status(wsp)}
        del dHp, qsets, wsp
        torch.cuda.empty_cache()

    result = {
        "metric": METRIC, "value": value, "unit": "TOPS", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "u8 codes (fp16 carriers, exact int accumulation); f32 in/out",
        "data": "synthetic (seeded; shapes and value distributions of the workload)",
        "config": {"workload": WORKLOAD, "quantizer": "Q_b2=BHQ-5 block16, Q_b1=PTQ-8 stochastic, X~/W~=PTQ-8",
                   "N": N, "C": C, "D": D, "global_batch": 128 * world,
                   "parallelism": f"replicas x{world} (independent batches)",
                   "l2": "flushed between timed steps (256 MiB write)",
                   "launch": ("eager C-ABI calls" if args.eager else
                              "one CUDA graph per call, captured from the C-ABI calls"),
                   "wall_s": t_wall},
        "per_call_ms": {k: float(v) for k, v in zip(names, per_call)},
        "per_call_gbs": {k: float(v) for k, v in call_gbs.items()},
        "quantizer_gbs": quant_gbs,
        "roofline": {"bound": "hbm", "kernel": kern_of[dom], "call": dom,
                     "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "peak_source": peak_src,
                     "algorithmic_bytes": alg_bytes[dom],
                     "traffic": traffic},
        "clocks": clk.summary(),
        "e2e": e2e,
        "forward": fwd,
        "adaptive_bhq": ada,
        "shift_quantizer": shf,
        "implicit_im2col": imp,
        "other_workloads": others,
        "paper_overhead_shape": ovh,
        "resnet50_sweep": sweep,
        "gpu_launches": int(sum(launches_per_call) * args.steps),
        "device_status": status,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(args.cpu_rows)
        if ovh is not None:
            # the paper timed its CPU quantizer routines on this shape (Sec.
            # 4.3); the oracle's whole gradient quantizers on one core beside it
            ovh["oracle_cpu_ms"] = oracle_overhead_shape()
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.destroy_process_group()


def _oracle_step(L, rows: int, seed: int):
    """One oracle pass over the first `rows` rows (the whole hot path)."""
    import oracle as orc
    dH, X = L.dH[:rows], L.X[:rows]
    orc.linear_backward(dH, X, L.W, KIND, BITS, BLOCK, seed)
    return 2 * 2 * rows * L.C * L.D


def cpu_baseline(rows: int):
    from paper_2010_14298_gb300 import workloads as wl
    import oracle
    oracle.build()
    L = wl.config(CONFIG_INDEX, batch=max(1, rows // 1024))[0]
    rows = L.N
    t = time.perf_counter()
    ops = _oracle_step(L, rows, 0)
    dt = time.perf_counter() - t
    return {"value": ops / dt / 1e12, "unit": "TOPS", "cores": 1, "kind": "oracle",
            "sample": f"{rows} im2col rows (batch {rows // 1024}) of the workload, "
                      f"full hot path, {dt:.1f} s single-threaded"}


def oracle_overhead_shape():
    """The oracle's gradient quantizers (range, scales / transform, SR, sums;
    Q_b2 only) on the paper's overhead shape, dH 401408 x 64, one core."""
    import oracle as orc
    from paper_2010_14298_gb300 import workloads as wl
    orc.build()
    dH = wl.random_grad(wl.rng(480), 128 * 56 * 56, 64, sigma=2.0, outlier_frac=0.01)
    out = {}
    for name, kind, bits, block in (("PTQ-8", orc.PTQ, 8, 0), ("PSQ-8", orc.PSQ, 8, 0),
                                    ("BHQ-5 block 16", orc.BHQ, 5, 16)):
        t = time.perf_counter()
        orc.quantize_grad(dH, kind, bits, block, 0, orc.STREAM_B2)
        out[name] = (time.perf_counter() - t) * 1e3
    return out


def run_reference(args):
    world, rank, _ = _dist()
    if rank != 0:
        return
    from paper_2010_14298_gb300 import workloads as wl
    import oracle
    oracle.build()
    L = wl.config(CONFIG_INDEX, batch=max(1, args.ref_rows // 1024))[0]
    rows = L.N
    for i in range(args.warmup):
        _oracle_step(L, min(rows, 1024), i)
    t = time.perf_counter()
    ops = 0
    for i in range(args.steps):
        ops += _oracle_step(L, rows, 100 + i)
    dt = time.perf_counter() - t
    value = ops / dt / 1e12
    out = {"impl": "reference", "metric": METRIC, "value": value, "unit": "TOPS",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": dt / args.steps * 1e3, "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64 oracle (f32 codes)",
           "data": "synthetic (seeded)",
           "config": {"workload": WORKLOAD, "sample_rows": rows},
           "cpu_baseline": {"value": value, "unit": "TOPS", "cores": 1,
                            "kind": "oracle",
                            "sample": f"{rows} im2col rows per step, full hot path"},
           "e2e": {"value": value, "unit": "TOPS", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--e2e-copy-streams", type=int, default=1,
                    help="streams per copy direction in the end-to-end pipeline")
    ap.add_argument("--cpu-rows", type=int, default=65536,
                    help="rows of the CPU-baseline sample (about 10 s of oracle work)")
    ap.add_argument("--ref-rows", type=int, default=8192,
                    help="rows per reference-arm step")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--forward-steps", type=int, default=50,
                    help="timed calls of the quantized forward GEMM (0: skip)")
    ap.add_argument("--adaptive-steps", type=int, default=50,
                    help="timed steps of the adaptive BHQ groups (0: skip)")
    ap.add_argument("--shift-steps", type=int, default=50,
                    help="timed steps of the shift quantizer path (0: skip)")
    ap.add_argument("--implicit-steps", type=int, default=50,
                    help="timed steps with the implicit im2col X operand (0: skip)")
    ap.add_argument("--sweep-steps", type=int, default=5,
                    help="timed rounds per layer of the ResNet-50 sweep (0: skip)")
    ap.add_argument("--config-steps", type=int, default=20,
                    help="timed steps of the other full-size workloads and of the paper's "
                         "overhead shape (0: skip)")
    ap.add_argument("--eager", action="store_true",
                    help="time the C-ABI calls directly instead of graph replays")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "native":
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_gpu(args)


if __name__ == "__main__":
    main()
