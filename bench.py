"""Benchmark: rounds of Efficient-Adam's two-way quantized error-feedback pipeline on one GB300.

One step = one full round: n worker compresses (Algorithm 2), the server step (Algorithm 1) and
x <- x - Q_s(w), on the default workload c5 (d = 1,558,000,000 fp32 parameters, n = 8 workers,
1-bit scaled sign with 4096-block scales, Adam moments on the workers).  The metric is round
throughput in parameter x worker elements per second.  Inputs are synthetic and resident in HBM
(the working set, ~213 GB, is far larger than the 129 MB L2, so no flush is needed between steps).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload c5] [--placement worker|server]
    python bench.py --impl reference     # the oracle on the host cores, same metric

With torchrun (N > 1) every rank runs an independent replica of the workload on its own GPU (the
simulated round does not shard: replicas only); the value is the sum of elements over all ranks
divided by the slowest rank's time.
"""
from __future__ import annotations

import argparse
import hashlib
import re
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "round throughput (param x worker elems/s) and achieved HBM GB/s vs GB300 peak"
UNIT = "param*worker elems/s"


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


_OVERRIDE = {}


def _workload(name: str):
    from paper_2205_14473_gb300 import workloads as W

    w = W.WORKLOADS[name]
    return w.with_(**_OVERRIDE) if _OVERRIDE else w


def _describe(w, placement: int) -> str:
    from paper_2205_14473_gb300 import workloads as W

    kinds = {W.Q_SIGN_L1: "1-bit scaled sign", W.Q_UNIFORM_MAX: "uniform grid", W.Q_POW2: "power-of-two",
             W.Q_IDENTITY: "identity"}

    def q(s):
        g = "whole-vector" if s.group == 0 else (f"{s.group}-block" if s.group > 0 else "per-tensor")
        extra = f" {s.bits}-bit{' stochastic' if s.stochastic else ''}" if s.kind == W.Q_UNIFORM_MAX else ""
        return f"{kinds[s.kind]}{extra}, {g} scales"
    where = "Adam at workers (Algorithm 2)" if placement == 0 else "Adam at server"
    return f"{w.name}: d={w.d:,} fp32, n={w.n} workers; Q_w {q(w.qw)}; Q_s {q(w.qs)}; {where}"


def algorithmic_bytes(w, placement: int) -> dict:
    """Bytes per launch that each kernel must move at least (fp32 state, codes at b bits)."""
    d, n = w.d, w.n
    bw, bs = w.qw.bits / 8.0, w.qs.bits / 8.0
    gw = 0 if w.qw.kind in (0, 3) else (1 if w.qw.group == 0 else (-(-d // w.qw.group) if w.qw.group > 0 else
                                                                    len(w.qw.segments)))
    gs = 0 if w.qs.kind in (0, 3) else (1 if w.qs.group == 0 else (-(-d // w.qs.group) if w.qs.group > 0 else
                                                                    len(w.qs.segments)))
    if placement == 0:
        compress = d * (16 + 12 + bw) + 4 * gw      # g, m, v, e read; m, v, e written; codes + scales
        server = d * (n * bw + 8 + bs) + 4 * (n * gw + gs)
    else:
        compress = d * (8 + 4 + bw) + 4 * gw        # g, e read; e written
        server = d * (n * bw + 24 + bs) + 4 * (n * gw + gs)
    apply = d * (8 + bs) + 4 * gs
    return {"compress": compress, "server": server, "apply": apply,
            "round": n * compress + server + apply}


_COMMENT = re.compile(r"//[^\n]*|/\*.*?\*/", re.S)


def _kernel_source_hash() -> str:
    """Hash of the CUDA sources with their comments removed: ncu figures taken on one version of
    the kernels stay valid across edits that change comments only."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2205_14473_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, f), encoding="utf-8") as fh:
            code = _COMMENT.sub("", fh.read())
        h.update(f.encode() + "\n".join(ln.rstrip() for ln in code.splitlines() if ln.strip()).encode())
    return h.hexdigest()[:16]


def _ncu_traffic(kernel: str, workload: str, placement: int):
    """Per-launch DRAM bytes of `kernel` from the committed ncu summary, if it was taken on the
    current kernel sources (profiles/ncu_traffic.txt: `kernel workload placement source-hash bytes`)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    if not os.path.exists(path):
        return None
    cur = _kernel_source_hash()
    for line in open(path):
        p = line.split()
        if len(p) == 5 and not line.startswith("#") and p[0] == kernel and p[1] == workload and \
                p[2] == str(placement) and p[3] == cur:
            return float(p[4])
    return None


# The kernels behind each step of a round (the finalize launches, which move a few KB, are left out).
ROLE_KERNELS = {"compress": ("worker_kernel", "worker_grouped", "worker_lazy", "encode_kernel"),
                "server": ("server_staged", "server_grouped", "server_lazy", "server_kernel"),
                "apply": ("apply_kernel",)}


def _ncu_traffic_role(role: str, workload: str, placement: int):
    """Summed per-launch DRAM bytes of the kernels that make up one step of a round, from the
    committed ncu summary, if every such row was taken on the current kernel sources."""
    vals = [_ncu_traffic(k, workload, placement) for k in ROLE_KERNELS[role]]
    vals = [v for v in vals if v is not None]
    return sum(vals) if vals else None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.samples = []
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "100"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None
        return self

    def _read(self):
        for line in self.proc.stdout:
            p = [x.strip() for x in line.split(",")]
            if len(p) >= 9:
                self.samples.append(p)

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.samples:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(p[1]) for p in self.samples if p[1].replace(".", "").isdigit()]
        mx = [float(p[2]) for p in self.samples if p[2].replace(".", "").isdigit()]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for p in self.samples:
            for name, v in zip(names, p[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(self.samples)}


# ------------------------------------------------------------------------------- CPU baseline

class OracleSample:
    """The oracle, as it stands, on a bounded sample of the workload: `blocks` whole 4096-blocks of
    every worker when the scales are per 4096-block (the round is separable by block; the global
    coordinates key the Philox counters), else a prefix of d with the same quantizers.  One step()
    is one full round (n worker steps, the server step, the update of x) on `threads` host threads
    (the workers, and chunks of whole scale groups, run concurrently)."""

    def __init__(self, w, placement: int, blocks: int = 16, threads: int = 1):
        import numpy as np

        import oracle as O
        from paper_2205_14473_gb300 import workloads as W

        if w.qw.group == 4096 and w.qs.group == 4096:
            sel = W.sample_blocks(w, blocks)
            lens = np.array([min(4096, w.d - b * 4096) for b in sel], np.int64)
            d = int(lens.sum())
            offs = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
            gidx = np.concatenate([np.arange(b * 4096, b * 4096 + l) for b, l in zip(sel, lens)])
            self.sample = f"{len(sel)} of {-(-w.d // 4096):,} 4096-blocks x {w.n} workers per round"
        else:
            d = min(w.d, blocks * 4096)
            offs, gidx = None, None
            self.sample = f"the first {d:,} coordinates x {w.n} workers per round"

        def quant(s):
            if offs is not None and s.kind in (W.Q_SIGN_L1, W.Q_UNIFORM_MAX):
                o = offs
            else:
                o = O.group_offsets(d, s.group if 0 < s.group <= d else 0)
            return O.Quantizer(s.kind, s.bits, o, stochastic=s.stochastic, pow2_k=s.pow2_k, pow2_K=s.pow2_K)

        self.d, self.n = d, w.n
        self.orc = O.OracleRound(d, w.n, quant(w.qw), quant(w.qs), w.alpha, w.beta1, w.beta2, w.eps,
                                 seed=w.seed, mode=placement, gidx=gidx, threads=threads)
        self.threads = threads
        rng = np.random.default_rng(0)
        self.grads = [(rng.standard_normal(d) * w.grad_std).astype(np.float32) for _ in range(w.n)]
        self.x = np.zeros(d, np.float32)

    def step(self):
        self.orc.compress_all(self.grads)
        self.orc.server_step()
        self.orc.apply(self.x)

    @property
    def units_per_step(self) -> int:
        return self.n * self.d


def host_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def _oracle_rate(w, placement: int, seconds: float, blocks: int, threads: int):
    ob = OracleSample(w, placement, blocks, threads)
    ob.step()  # warm-up (page-in of the sample's arrays)
    rounds, t0 = 0, time.perf_counter()
    while True:
        ob.step()
        rounds += 1
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    return rounds * ob.units_per_step / el, f"{ob.sample}; {rounds} rounds in {el:.1f} s"


def cpu_baseline(w, placement: int, seconds: float = 12.0):
    """The oracle, as it stands, on a bounded sample of the workload, timed on this host's cores:
    one thread per worker (n threads: the workers concurrently, then the server step and the update
    of x over chunks of whole scale groups), and on one core for comparison."""
    cores = host_cores()
    threads = max(1, min(w.n, cores))
    val, sample = _oracle_rate(w, placement, seconds / 2, 1024, threads)
    val1, sample1 = _oracle_rate(w, placement, seconds / 2, 128, 1)
    return {"value": val, "unit": UNIT, "cores": threads, "threads": threads, "cores_available": cores,
            "kind": "oracle", "sample": f"{sample}, {threads} host threads (one per worker)",
            "value_1core": val1, "sample_1core": f"{sample1}, one host thread"}


# ---------------------------------------------------------------------------------- GPU bench

def max_over_ranks(ms: float, world: int, device) -> float:
    """The job's time: the slowest rank's timed region (an all-reduce MAX when world > 1)."""
    if world <= 1:
        return ms
    import torch

    t = torch.tensor([ms], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(n: int, d: int, steps: int, world: int, t_max_ms: float) -> float:
    """Whole-job parameter x worker elements per second: every rank runs its own replica of the
    n-worker round on d coordinates (weak scaling), so the job processes n d steps world units."""
    return n * d * steps * world / (t_max_ms / 1e3)


NOMINAL_HBM_GBS = 8000.0  # the GB300's nominal ~8 TB/s, the reference of the 70% target


class RoundTimer:
    """A workload's round state on one device (library handle with its workspace, n resident
    gradients, x) and CUDA-event timing of its rounds on the library's stream."""

    def __init__(self, w, placement: int, dev, stream):
        import torch

        import paper_2205_14473_gb300 as ea
        from paper_2205_14473_gb300 import workloads as W

        self.w, self.placement, self.dev, self.stream = w, placement, dev, stream
        cfg = ea.EAConfig.from_workload(w, placement=placement)
        with torch.cuda.stream(stream):
            self.rnd = ea.EARound(cfg, stream=stream, device=dev)
            self.grads = [torch.empty(w.d, dtype=torch.float32, device=dev) for _ in range(w.n)]
            for i, g in enumerate(self.grads):
                W.gradient_device(w, i, 0, g)
            self.x = torch.zeros(w.d, dtype=torch.float32, device=dev)
        stream.synchronize()

    def one_round(self, ev=None):
        w, rnd, s = self.w, self.rnd, self.stream
        for i in range(w.n):
            if ev is not None:
                ev["c0"][i].record(s)
            rnd.worker_compress(i, self.grads[i])
            if ev is not None:
                ev["c1"][i].record(s)
        if ev is not None:
            ev["s0"].record(s)
        rnd.server_step()
        if ev is not None:
            ev["s1"].record(s)
        rnd.apply(self.x)
        if ev is not None:
            ev["a1"].record(s)

    def run(self, steps: int, warmup: int, barrier=lambda: None, clocks=None):
        """warmup untimed rounds, then `steps` rounds between two events (per-kernel events inside);
        returns (total ms, per-launch ms lists)."""
        import torch

        for _ in range(warmup):
            self.one_round()
        self.stream.synchronize()
        E = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
        per = [{"c0": [E() for _ in range(self.w.n)], "c1": [E() for _ in range(self.w.n)], "s0": E(), "s1": E(),
                "a1": E()} for _ in range(steps)]
        start, end = E(), E()
        if clocks is not None:
            time.sleep(0.3)
        barrier()
        torch.cuda.synchronize(self.dev)
        start.record(self.stream)
        for k in range(steps):
            self.one_round(per[k])
        end.record(self.stream)
        torch.cuda.synchronize(self.dev)
        barrier()
        comp = [ev["c0"][i].elapsed_time(ev["c1"][i]) for ev in per for i in range(self.w.n)]
        serv = [ev["s0"].elapsed_time(ev["s1"]) for ev in per]
        appl = [ev["s1"].elapsed_time(ev["a1"]) for ev in per]
        self.rnd.sync()
        return start.elapsed_time(end), comp, serv, appl

    def kernel_figures(self, ms_total: float, steps: int, comp, serv, appl) -> dict:
        """Per-kernel mean times and algorithmic GB/s, against the measured copy peak and 8 TB/s."""
        ab = algorithmic_bytes(self.w, self.placement)
        peak, _ = _peaks()
        out = {"workload": self.w.name, "placement": "worker" if self.placement == 0 else "server",
               "d": self.w.d, "n_workers": self.w.n, "steps": steps, "ms_per_round": ms_total / steps,
               "elems_per_s": self.w.n * self.w.d * steps / (ms_total / 1e3)}
        for name, ts in (("compress", comp), ("server", serv), ("apply", appl)):
            ms = statistics.mean(ts)
            gbs = ab[name] / (ms / 1e3) / 1e9
            out[name] = {"ms": ms, "min_ms": min(ts), "gbs": gbs, "frac_measured": gbs / peak,
                         "frac_8tbs": gbs / NOMINAL_HBM_GBS, "bytes": ab[name],
                         "traffic": _ncu_traffic_role(name, self.w.name, self.placement)}
        rgbs = ab["round"] / (ms_total / steps / 1e3) / 1e9
        out["round"] = {"gbs": rgbs, "frac_measured": rgbs / peak, "frac_8tbs": rgbs / NOMINAL_HBM_GBS,
                        "bytes": ab["round"]}
        return out

    def free(self):
        import torch

        self.rnd = self.grads = self.x = None
        torch.cuda.synchronize(self.dev)
        torch.cuda.empty_cache()


# The other workloads and placements timed after the headline line (each alone on the device, its
# workspace freed before the next): the placement trade-off and the per-kernel rates at c3 and c4.
EXTRA_CONFIGS = [("c5", 1), ("c4", 0), ("c4", 1), ("c3", 0), ("c3", 1)]


def run_gpu(args, rank: int, world: int, local_rank: int):
    import torch

    from paper_2205_14473_gb300 import build as B

    B.build()
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    w = _workload(args.workload)
    placement = 0 if args.placement == "worker" else 1
    stream = torch.cuda.Stream(dev)
    rt = RoundTimer(w, placement, dev, stream)
    barrier = (lambda: torch.distributed.barrier()) if world > 1 else (lambda: None)
    with ClockSampler(local_rank) as clk:
        ms_total, comp, serv, appl = rt.run(args.steps, args.warmup, barrier, clocks=clk)
    figs = rt.kernel_figures(ms_total, args.steps, comp, serv, appl)

    # ---- end to end through the C-ABI with host buffers (pinned gradients read over the host link,
    # the broadcast message read back every step)
    e2e = None
    if not args.no_e2e:
        e2e = run_e2e(args, w, rt.rnd, rt.x, dev, stream)
    rnd_ws = rt.rnd.workspace_bytes
    launches = rt.rnd.launches_per_round
    rt.free()

    t_max = max_over_ranks(ms_total, world, dev)
    value = job_throughput(w.n, w.d, args.steps, world, t_max)
    ab = algorithmic_bytes(w, placement)
    peak, peak_kind = _peaks()
    comp_ms = figs["compress"]["ms"]
    achieved = ab["compress"] / (comp_ms / 1e3) / 1e9
    traffic = _ncu_traffic("worker_kernel", w.name, placement)
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": t_max / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": _describe(w, placement), "d": w.d, "n_workers": w.n, "global_batch": None,
                   "seq_len": None, "parallelism": f"replicas{world}" if world > 1 else "single GPU",
                   "l2": "inputs larger than L2 (working set %.0f GB)" % ((rnd_ws + (w.n + 1) * w.d * 4) / 1e9),
                   "placement": "worker" if placement == 0 else "server"},
        "roofline": {"bound": "hbm", "kernel": "worker_kernel (compress)", "achieved": achieved, "peak": peak,
                     "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak, "traffic": traffic,
                     "algorithmic_bytes_per_launch": ab["compress"],
                     "peak_nominal": NOMINAL_HBM_GBS, "frac_nominal": achieved / NOMINAL_HBM_GBS,
                     "note": "peak = the driver-measured copy bandwidth (a torch copy), which a streaming "
                             "kernel can exceed; frac_nominal is against the GB300's nominal ~8 TB/s"},
        "kernels_ms": {"compress_mean": comp_ms, "compress_min": figs["compress"]["min_ms"],
                       "server_mean": figs["server"]["ms"], "apply_mean": figs["apply"]["ms"],
                       "server_gbs": figs["server"]["gbs"], "apply_gbs": figs["apply"]["gbs"],
                       "round_gbs": figs["round"]["gbs"],
                       "server_frac_8tbs": figs["server"]["frac_8tbs"],
                       "compress_frac_8tbs": figs["compress"]["frac_8tbs"]},
        "gpu_launches": launches * args.steps,
        "clocks": clk.summary(),
        "e2e": e2e,
    }
    if not args.no_extra and world == 1 and not _OVERRIDE:
        extra = {}
        for name, pl in EXTRA_CONFIGS:
            if (name, pl) == (w.name, placement):
                continue
            we = _workload(name)
            rte = RoundTimer(we, pl, dev, stream)
            with ClockSampler(local_rank) as clk2:
                ms, c, sv, ap = rte.run(args.extra_steps, max(3, args.warmup), clocks=clk2)
            f = rte.kernel_figures(ms, args.extra_steps, c, sv, ap)
            f["clocks"] = clk2.summary()
            f["gpu_launches"] = rte.rnd.launches_per_round * args.extra_steps
            extra[f"{name}/{'W' if pl == 0 else 'S'}"] = f
            rte.free()
        out["configs"] = extra
    return out


def run_e2e(args, w, rnd, x, dev, stream):
    """The same rounds through the C-ABI with every gradient in pinned host memory.  The compress
    kernel reads it straight over the host link (pinned memory is mapped into the GPU's address
    space), and the broadcast message (codes + scales, the round's output) is read back into pinned
    host memory.  For comparison, the same rounds with copy-engine H2D copies into two device
    buffers that overlap the previous worker's compress, and the copies alone."""
    import torch

    import paper_2205_14473_gb300 as ea

    avail = 0
    try:
        for line in open("/proc/meminfo"):
            if line.startswith("MemAvailable:"):
                avail = int(line.split()[1]) * 1024
    except Exception:
        pass
    gbytes = w.d * 4
    n_host = w.n
    while n_host > 1 and n_host * gbytes > 0.3 * avail:
        n_host //= 2
    host = [torch.empty(w.d, dtype=torch.float32, pin_memory=True) for _ in range(n_host)]
    gen = torch.Generator().manual_seed(w.seed)
    for h in host:
        h.normal_(0.0, w.grad_std, generator=gen)
    codes, scales = rnd.view(ea.EA_VIEW_CODES_SERVER), rnd.view(ea.EA_VIEW_SCALES_SERVER)
    codes_h = torch.empty(codes.numel(), dtype=codes.dtype, pin_memory=True)
    scales_h = torch.empty(max(scales.numel(), 1), dtype=scales.dtype, pin_memory=True)
    d2h = codes.numel() * codes.element_size() + scales.numel() * scales.element_size()
    nstage = 2
    staging = [torch.empty(w.d, dtype=torch.float32, device=dev) for _ in range(nstage)]
    copy = torch.cuda.Stream(dev)
    ev_copied = [torch.cuda.Event() for _ in range(nstage)]
    ev_used = [torch.cuda.Event() for _ in range(nstage)]

    def read_back():
        with torch.cuda.stream(stream):
            codes_h.copy_(codes, non_blocking=True)
            if scales.numel():
                scales_h[: scales.numel()].copy_(scales, non_blocking=True)

    def step_direct():
        for i in range(w.n):
            ea.ea_worker_compress(rnd.h, i, host[i % n_host].data_ptr())
        ea.ea_server_step(rnd.h)
        ea.ea_worker_apply(rnd.h, x.data_ptr())
        read_back()

    def step_staged():
        for i in range(w.n):
            b = i % nstage
            with torch.cuda.stream(copy):
                copy.wait_event(ev_used[b])
                staging[b].copy_(host[i % n_host], non_blocking=True)
                ev_copied[b].record(copy)
            stream.wait_event(ev_copied[b])
            ea.ea_worker_compress(rnd.h, i, staging[b].data_ptr())
            ev_used[b].record(stream)
        ea.ea_server_step(rnd.h)
        ea.ea_worker_apply(rnd.h, x.data_ptr())
        read_back()

    def timed(fn):
        for _ in range(max(1, args.warmup)):
            fn()
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        for _ in range(args.steps):
            fn()
        torch.cuda.synchronize(dev)
        return time.perf_counter() - t0

    el = timed(step_direct)
    el_staged = timed(step_staged)
    t1 = time.perf_counter()
    with torch.cuda.stream(copy):
        for i in range(w.n):
            staging[i % nstage].copy_(host[i % n_host], non_blocking=True)
    torch.cuda.synchronize(dev)
    h2d_only = time.perf_counter() - t1
    return {"value": w.n * w.d * args.steps / el, "unit": UNIT, "h2d_bytes_per_step": w.n * gbytes,
            "d2h_bytes_per_step": d2h, "ms_per_step": el / args.steps * 1e3, "host_buffers": n_host,
            "staged_copy_ms_per_step": el_staged / args.steps * 1e3,
            "h2d_copy_only_ms_per_step": h2d_only * 1e3, "h2d_copy_gbs": w.n * gbytes / h2d_only / 1e9,
            "note": "ea_worker_compress/ea_server_step/ea_worker_apply with every gradient in pinned host memory, "
                    "read by the compress kernel over the host link each step, and the broadcast message read back"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ea", choices=["ea", "reference"])
    ap.add_argument("--workload", default="c5")
    ap.add_argument("--placement", default="worker", choices=["worker", "server"])
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--d", type=int, default=None, help="override d (small profiling cases)")
    ap.add_argument("--n", type=int, default=None, help="override the worker count")
    ap.add_argument("--no-extra", action="store_true", help="time the headline workload only")
    ap.add_argument("--extra-steps", type=int, default=10, help="timed rounds of each extra workload")
    args = ap.parse_args()

    if args.d:
        _OVERRIDE["d"] = args.d
    if args.n:
        _OVERRIDE["n"] = args.n
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    w = _workload(args.workload)
    placement = 0 if args.placement == "worker" else 1

    if args.impl == "reference":
        # the oracle on the host cores, same workload/metric; under torchrun only rank 0 runs
        if rank != 0:
            return
        import oracle

        oracle.build()
        cores = host_cores()
        threads = max(1, min(w.n, cores))
        ob = OracleSample(w, placement, blocks=1024, threads=threads)
        for _ in range(args.warmup):
            ob.step()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            ob.step()
        el = time.perf_counter() - t0
        val = args.steps * ob.units_per_step / el
        cb = {"value": val, "unit": UNIT, "cores": threads, "threads": threads, "cores_available": cores,
              "kind": "oracle",
              "sample": f"{ob.sample}; {args.steps} timed rounds in {el:.2f} s, {threads} host threads (one per worker)"}
        out = {"impl": "reference", "metric": METRIC, "value": val, "unit": UNIT, "n_gpus": 1,
               "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
               "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
               "data": "synthetic", "config": {"workload": _describe(w, placement), "d": w.d, "n_workers": w.n},
               "cpu_baseline": cb, "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0,
                                           "d2h_bytes_per_step": 0}}
        print(json.dumps(out), flush=True)
        return

    if world > 1:
        import torch

        torch.distributed.init_process_group("nccl")
    out = run_gpu(args, rank, world, local_rank)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle

        oracle.build()
        out["cpu_baseline"] = cpu_baseline(w, placement, seconds=args.cpu_seconds)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch

        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
