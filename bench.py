#!/usr/bin/env python3
"""Throughput of the Hier-AVG hot path on GB300.

One bench "step" is one global round of Algorithm 1 (Sec. 3.1): K2 x (K1 local
SGD steps of all P learners + a local average) + the global average, on
synthetic Gaussian-mixture data already resident in HBM.  The metric is
learner-samples per second (P * B * K1 * K2 per round).

  python bench.py [--gpus N --steps K --warmup W] [--workload mlp4096|mlp2048|mlp512|softmax]
  python bench.py --impl reference ...   # the CPU oracle on a bounded sample
  python bench.py --sweep [--sweep-D D ...]   # averaging-only sweep (P = 128), GB/s table

The default workload is the largest one that fits one GPU: 32 learners of the
ImageNet-shaped MLP 12288 -> 4096 -> 4096 -> 1000 (about 71M parameters each).

Under torchrun (N > 1) every rank runs an independent replica on its own GPU
(the learners of one replica never leave their GPU), timing is max over ranks
and ``value`` is the sum over replicas ("scaling": "weak").
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "learner-samples/s per Hier-AVG round"
UNIT = "learner-samples/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 512 << 20
DOM_SAMPLE = 7   # time about 1 in 7 launches of the dominant kernel (see dom_sample)


def dom_sample(per_round: int) -> int:
    """The sampling interval: the smallest n >= DOM_SAMPLE coprime with the dominant
    kernel's launches per round, so that the timed launches cycle through every position
    in the round (the first step of a block reads the cluster means and runs faster)."""
    n = DOM_SAMPLE
    while math.gcd(n, max(1, per_round)) != 1:
        n += 1
    return n


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mlp4096")
    ap.add_argument("--sweep", action="store_true")
    ap.add_argument("--sweep-D", type=int, nargs="+", default=None,
                    help="parameter counts of the sweep (default: 1M, 11.2M, 32M, 64M)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-sweep-point", action="store_true",
                    help="skip the averaging-only point (P = 128, D = 64M) in the JSON line")
    ap.add_argument("--N", type=int, default=None,
                    help="samples per learner (default: the workload's); for small profiling runs")
    ap.add_argument("--P", type=int, default=None,
                    help="learners (default: the workload's; a multiple of S); for small profiling runs")
    return ap.parse_args()


def dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def job_seconds(seconds: float, ws: int, device=None) -> float:
    """The job's time: the maximum over the ranks of each rank's timed seconds
    (every rank runs an independent replica; the slowest one ends the job)."""
    if ws <= 1:
        return seconds
    import torch
    import torch.distributed as dist
    t = torch.tensor([seconds], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(ws: int, units_per_round: int, rounds: int, seconds: float) -> float:
    """Whole-job throughput: the units all replicas processed over the job's time."""
    return ws * units_per_round * rounds / seconds


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 20 ms."""
    Q = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                       "-lms", "20"], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        self.marks = []

    def mark(self):
        self.marks.append(time.time())

    def stop(self, uuid: str | None):
        if self.p is None:
            return None
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        rows = []
        with open(self.f.name) as fh:
            for line in fh:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 10:
                    continue
                rows.append(parts)
        os.unlink(self.f.name)
        if uuid:
            mine = [r for r in rows if uuid in r[1]]
            rows = mine or rows
        if not rows:
            return None

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[2]) for r in rows if num(r[2]) is not None]
        mx = [num(r[3]) for r in rows if num(r[3]) is not None]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for n, v in zip(names, r[6:10]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(rows),
                "power_w_max": max((num(r[4]) or 0) for r in rows)}


def src_hash(*names):
    h = hashlib.sha256()
    for n in names:
        with open(os.path.join(ROOT, "paper_1903_05133_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(kind: str, workload: str, P: int):
    """DRAM bytes per launch of a kernel from a committed ncu summary, if the kernel
    source has not changed since it was captured.  A capture taken with fewer
    learners (``captured_P``) is scaled to P: every learner's weights are streamed
    once per launch, so the bytes grow in proportion to the learners."""
    p = os.path.join(ROOT, "profiles", "ncu_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    e = d.get(workload, {}).get(kind)
    if not e:
        return None
    if e.get("source_hash") != src_hash(*e.get("sources", [])):
        return None
    by = e.get("dram_bytes_per_launch")
    cp = e.get("captured_P")
    return by * P / cp if (by is not None and cp) else by


def run_config(w, ws: int) -> dict:
    """The workload as both arms of the bench name it."""
    return {"workload": w.name, "P": w.P, "S": w.S, "K1": w.K1, "K2": w.K2, "B": w.B,
            "dims": list(w.dims), "lr": w.lr, "N": w.N,
            "parallelism": f"{w.P} simulated learners per GPU" + (f" x {ws} replicas" if ws > 1 else ""),
            "l2": f"GPU arm: flushed between timed rounds ({L2_FLUSH_BYTES >> 20} MB write, untimed); "
                  f"parameters {w.P * w.n_params * 4 / 1e9:.2f} GB",
            "master": "fp32", "gemm_operands": w.precision}


# ----------------------------------------------------------------------------- oracle
def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


class OracleSample:
    """The CPU oracle, as it stands, on a bounded sample of a Hier-AVG round.

    A round is P * K1 * K2 learner steps plus K2 local averages of P / S clusters and
    one global average.  One sample times ``steps`` local SGD steps of one learner
    (learner 0, on its own data, batches read as in the round) and the local average
    of one cluster of S learners over a 1 / ``avg_split`` slice of the parameter row.
    The round's time is extrapolated from them: the learner steps times P * K1 * K2,
    the cluster average (times avg_split) times K2 * P / S, and the global average
    as (P - 1) / (S - 1) cluster averages (a tree over P rows instead of S)."""

    def __init__(self, w, X0, y0, layers):
        import numpy as np
        import oracle
        self.w = w
        self.mode = "fp32" if w.precision == "fp32" else "bf16"
        params = []
        for Wl, bl in layers:
            params += [Wl.numpy()[None].copy(), bl.numpy()[None].copy()]
        prob = oracle.MLPProblem(X0.float().numpy(), y0.numpy().astype(np.int64), w.B,
                                 len(w.dims) - 1, self.mode)
        self.learner = oracle.HierAvgOracle(1, 1, w.K1, w.K2, w.lr, prob, params, self.mode)
        D = w.n_params
        self.avg_split = 8 if D * w.S * 4 > (1 << 30) else 1
        cols = -(-D // self.avg_split)
        rng = np.random.default_rng(0)
        self.cluster = rng.standard_normal((w.S, cols), dtype=np.float32)
        self.steps = 1 if D > 10_000_000 else w.K1

    def run(self):
        """One sample: (seconds of the learner steps, seconds of the slice average)."""
        import oracle
        t0 = time.perf_counter()
        for _ in range(self.steps):
            self.learner.step()
        t1 = time.perf_counter()
        oracle.local_average(self.cluster, self.w.S)
        t2 = time.perf_counter()
        return t1 - t0, t2 - t1

    def round_seconds(self, t_steps: float, t_avg: float) -> float:
        w = self.w
        per_step = t_steps / self.steps
        per_cluster_avg = t_avg * self.avg_split
        avgs = w.K2 * (w.P // w.S) + (w.P - 1) / max(1, w.S - 1)
        return w.P * w.K1 * w.K2 * per_step + avgs * per_cluster_avg

    def describe(self) -> str:
        w = self.w
        frac = f"1/{self.avg_split} of the {w.n_params}-parameter row" if self.avg_split > 1 \
            else f"the whole {w.n_params}-parameter row"
        return (f"extrapolated: {self.steps} local SGD step(s) of one learner (B = {w.B}) and one local "
                f"average of {w.S} learners over {frac}, scaled to a round ({w.P * w.K1 * w.K2} learner "
                f"steps, {w.K2 * (w.P // w.S)} cluster averages, one global average counted as "
                f"(P-1)/(S-1) cluster averages); numpy, {self.mode} operands, float64 products, "
                f"multi-threaded BLAS")


def oracle_inputs_cpu(w, X0=None, y0=None):
    """Learner 0's data (generated on the CPU unless given) and the shared w0."""
    from paper_1903_05133_gb300.inputs import initial_layers, learner_data
    if X0 is None:
        X0, y0 = learner_data(w, learners=[0])
    return X0, y0, initial_layers(w)


def run_reference(args):
    """The CPU oracle timed as it stands on the host cores: every bench step is one
    bounded sample of the workload's round (OracleSample), and the value is the
    round's learner-samples over the extrapolated round time."""
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    from paper_1903_05133_gb300 import configs
    w = configs.SHORT[args.workload]
    X0, y0, layers = oracle_inputs_cpu(w)
    smp = OracleSample(w, X0, y0, layers)
    runs = [smp.run() for _ in range(args.warmup + args.steps)][args.warmup:]
    ts = statistics.mean(r[0] for r in runs)
    ta = statistics.mean(r[1] for r in runs)
    value = w.samples_per_round / smp.round_seconds(ts, ta)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000 * statistics.mean(a + b for a, b in runs),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16-operands/f64-products" if w.precision == "bf16" else "f32/f64-products",
            "data": "synthetic (seeded Gaussian mixture, CIFAR-10 / ImageNet shaped)",
            "config": run_config(w, ws),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                             "sample": smp.describe() + "; each bench step is one sample"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- ours
def gemm_report(by: float, fl: float, ms: float, hbm_gbs: float, tc_tflops: float) -> dict:
    """TFLOP/s of a set of launches against the tensor-core rate, next to the ceiling
    that the HBM roofline sets for their arithmetic intensity (flops per byte)."""
    tflops = fl / (ms / 1e3) / 1e12
    ceiling = min(tc_tflops, (fl / by) * hbm_gbs / 1e3) if by > 0 else tc_tflops
    return {"TFLOPs": round(tflops, 2), "tensor_frac": round(tflops / tc_tflops, 4),
            "flop_per_byte": round(fl / by, 2) if by > 0 else None,
            "hbm_bound_tensor_frac_ceiling": round(ceiling / tc_tflops, 4),
            "frac_of_hbm_bound_ceiling": round(tflops / ceiling, 4)}


def averaging_point(dev, flush, hbm_gbs: float) -> dict:
    """One point of the averaging-only sweep: P = 128 fp32 learner rows of D = 64M
    parameters (32.8 GB, far above L2), the local average over clusters of S = 8 and
    the fused last-local + global average; L2 flushed before every timed launch."""
    import torch
    from paper_1903_05133_gb300.hier_avg import local_average_buffer, local_global_average_buffer
    from paper_1903_05133_gb300.inputs import replica_matrix
    P, D, S = 128, 64_000_000, 8
    wm = replica_matrix(P, D, device=dev)
    out = {"P": P, "D": D, "S": S, "bytes_per_pass": 8.0 * P * D,
           "timing": "median of 7 launches, CUDA events, L2 flushed before each"}
    for op, fn in (("local", lambda: local_average_buffer(wm, S)),
                   ("local_global", lambda: local_global_average_buffer(wm, S))):
        fn()
        ms = []
        for _ in range(7):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            torch.cuda.synchronize()
            ms.append(a.elapsed_time(b))
        med = statistics.median(ms)
        gbs = 8.0 * P * D / (med / 1e3) / 1e9
        out[op] = {"ms": round(med, 4), "GBps": round(gbs, 1), "frac_of_measured_hbm": round(gbs / hbm_gbs, 4),
                   "frac_of_8TBps": round(gbs / 8000.0, 4)}
    del wm
    torch.cuda.empty_cache()
    return out



def run_ours(args):
    import torch
    import torch.distributed as dist
    from paper_1903_05133_gb300 import configs
    from paper_1903_05133_gb300.hier_avg import HierAvg
    from paper_1903_05133_gb300.inputs import initial_layers, learner_data

    ws, rank, local = dist_env()
    if ws > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = configs.SHORT[args.workload]
    if args.N:
        w = w.replace(N=args.N)
    if args.P:
        if args.P % w.S:
            raise SystemExit(f"--P must be a multiple of S = {w.S}")
        w = w.replace(P=args.P)
    X, y = learner_data(w, device=dev)
    X0c, y0c = X[:1].cpu(), y[:1].cpu()          # learner 0's data for the CPU oracle
    layers = initial_layers(w, device=dev)
    ha = HierAvg(w.P, w.S, w.K1, w.K2, w.lr, w.B, w.dims, w.precision)
    params = ha.pack(layers, device=dev)
    ha.bind(params, X, y)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    for _ in range(args.warmup):
        ha.round()
    ha.check()
    torch.cuda.synchronize()

    # Untimed profiling pass: every kernel kind, to find the dominant kernel and to
    # report the per-kind breakdown.  (An event pair around a launch separates it
    # from its neighbours, so the timed rounds below time only the dominant kind.)
    kinds = ["gather", "forward", "xent", "backward", "local_avg", "global_avg", "head",
             "update_forward"]
    ha.profile(True)
    for _ in range(max(1, min(args.steps, 3))):
        flush.zero_()
        ha.round()
    prof = {k: ha.profile_read(k) for k in kinds}
    ha.profile(False)
    main_kinds = ["forward", "backward", "local_avg", "global_avg", "xent", "gather", "head",
                  "update_forward"]
    dom = max(main_kinds, key=lambda k: prof[k].total_ms)

    props = torch.cuda.get_device_properties(dev)
    uuid = str(getattr(props, "uuid", "") or "")
    sampler = ClockSampler()
    time.sleep(0.05)
    # one launch in DOM_SAMPLE of the dominant kernel is timed (events separate it from
    # its neighbours; timing every launch cost ~9 % of the round at 3072-512-10)
    n_prof_rounds = max(1, min(args.steps, 3))
    sample = dom_sample(prof[dom].launches // n_prof_rounds)
    ha.profile([dom])
    ha.profile_every(sample)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    if ws > 1:
        dist.barrier()
    torch.cuda.synchronize()
    launches0 = ha.launches()
    for k in range(args.steps):
        flush.zero_()                      # L2 flushed between timed rounds (not timed)
        starts[k].record()
        ha.round()
        ends[k].record()
    torch.cuda.synchronize()
    gpu_launches = ha.launches() - launches0   # the library's own count of its kernel launches
    if ws > 1:
        dist.barrier()
    clocks = sampler.stop(uuid)
    ha.check()
    round_ms = [s.elapsed_time(e) for s, e in zip(starts, ends)]
    T = job_seconds(sum(round_ms) / 1000.0, ws, dev)
    per_round = w.samples_per_round
    value = replica_throughput(ws, per_round, args.steps, T)

    dom_live = ha.profile_read(dom)          # the dominant kernel, timed inside the timed rounds
    ha.profile(False)
    ha.profile_every(1)
    # the same rounds again without any per-kernel events (diagnostic, untimed)
    plain_ms = []
    for k in range(min(args.steps, 10)):
        flush.zero_()
        a_ev, b_ev = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a_ev.record()
        ha.round()
        b_ev.record()
        torch.cuda.synchronize()
        plain_ms.append(a_ev.elapsed_time(b_ev))
    pk, pk_src = peaks()
    hbm = pk["hbm_gbs"]
    tc = pk.get("bf16_tflops_sustained") or pk["bf16_tflops"]
    dom_ms, dom_n, dom_bytes, dom_flops = dom_live
    achieved = dom_bytes / (dom_ms / 1e3) / 1e9 if dom_ms > 0 else None
    kernels = {}
    total_ms = max(1e-9, sum(v.total_ms for v in prof.values()))
    for k in kinds:
        ms, n, by, fl = prof[k]
        if n and ms > 0:
            e = {"launches": n, "total_ms": round(ms, 4), "avg_us": round(1e3 * ms / n, 2),
                 "share": round(ms / total_ms, 4), "GBps": round(by / (ms / 1e3) / 1e9, 1)}
            if fl > 0 and k not in ("local_avg", "global_avg"):
                e.update(gemm_report(by, fl, ms, hbm, tc))
            kernels[k] = e
    avg_ms = prof["local_avg"].total_ms + prof["global_avg"].total_ms
    avg_by = prof["local_avg"].bytes + prof["global_avg"].bytes
    step_kinds = ("forward", "backward", "update_forward", "head")
    step_ms = sum(prof[k].total_ms for k in step_kinds)
    step_fl = sum(prof[k].flops for k in step_kinds)
    step_by = sum(prof[k].bytes for k in step_kinds)
    traffic = ncu_traffic(dom, w.name, w.P) if not (args.P or args.N) else None
    roofline = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": hbm,
                "unit": "GB/s", "frac": (achieved / hbm) if achieved else None,
                "peak_source": f"{pk_src} (HBM copy)",
                "traffic": traffic,
                "algorithmic_bytes_per_launch": dom_bytes / max(1, dom_n),
                "avg_launch_us": 1e3 * dom_ms / max(1, dom_n),
                "timing": f"CUDA events around every {sample}th launch of this kernel inside the timed rounds",
                "launches_timed": dom_n}
    if dom_flops > 0:
        roofline["tensor"] = gemm_report(dom_bytes, dom_flops, dom_ms, hbm, tc)
    l2_bytes = torch.cuda.get_device_properties(dev).L2_cache_size
    params_bytes = 4.0 * w.P * ha.ld

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000 * T / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.precision,
            "data": "synthetic (seeded Gaussian mixture, CIFAR-10 / ImageNet shaped)",
            "config": run_config(w, ws),
            "roofline": roofline,
            "gemm": dict(gemm_report(step_by, step_fl, step_ms, hbm, tc),
                         note="all learner-step kernels of a round (forward, backward, "
                              "update+forward, head) from the profiling pass; bf16 operands, "
                              "fp32 accumulate; tensor fractions of the measured sustained "
                              "bf16 dense rate"),
            "averaging": {"GBps": avg_by / (avg_ms / 1e3) / 1e9 if avg_ms > 0 else None,
                          "frac_of_measured_hbm": (avg_by / (avg_ms / 1e3) / 1e9 / hbm) if avg_ms > 0 else None,
                          "frac_of_8TBps": (avg_by / (avg_ms / 1e3) / 8e12) if avg_ms > 0 else None,
                          "l2_assisted": params_bytes <= l2_bytes,
                          "note": "in-round local and global averages; with all parameters "
                                  "smaller than L2 part of each average is served from L2"},
            "kernels": kernels,
            "kernels_timing": "untimed profiling pass before the timed rounds, events around every launch",
            "ms_per_step_without_kernel_events": statistics.median(plain_ms),
            "gpu_launches": gpu_launches,
            "clocks": clocks}

    # ---- end to end through the C ABI from pinned host memory
    if not args.no_e2e:
        Xh = X.cpu().pin_memory()
        yh = y.cpu().pin_memory()
        loss = torch.empty(w.P, dtype=torch.float32, pin_memory=True)
        for _ in range(max(1, args.warmup)):
            ha.round_host(Xh, yh, loss)
        if ws > 1:
            dist.barrier()
        torch.cuda.synchronize()
        # events on the handle's stream around every call: the device time of each
        # round from host memory, next to the host clock over all of them
        e_a = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        e_b = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
        t0 = time.perf_counter()
        for k in range(args.steps):
            e_a[k].record()
            ha.round_host(Xh, yh, loss)
            e_b[k].record()
        torch.cuda.synchronize()
        Te = job_seconds(time.perf_counter() - t0, ws, dev)
        dev_ms = sorted(a.elapsed_time(b) for a, b in zip(e_a, e_b))
        rows = w.B * w.K1 * w.K2
        es = 2 if w.precision == "bf16" else 4
        line["e2e"] = {"value": replica_throughput(ws, per_round, args.steps, Te), "unit": UNIT,
                       "h2d_bytes_per_step": w.P * rows * w.dims[0] * es + w.P * w.N * 4,
                       "d2h_bytes_per_step": w.P * 4,
                       "api": "hier_avg_round_host (pinned host X, y; loss read back)",
                       "ms_per_step": 1000 * Te / args.steps,
                       "device_ms_per_step_median": statistics.median(dev_ms),
                       "device_ms_per_step_max": dev_ms[-1]}
        del Xh, yh

    if rank == 0 and not args.no_sweep_point:
        del ha, params, X, y
        torch.cuda.empty_cache()
        line["averaging_sweep"] = averaging_point(dev, flush, hbm)

    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        X0, y0, lc = oracle_inputs_cpu(w, X0c, y0c)
        smp = OracleSample(w, X0, y0, lc)
        smp.run()                                           # warm-up sample
        ts, ta = smp.run()
        v = w.samples_per_round / smp.round_seconds(ts, ta)
        line["cpu_baseline"] = {"value": v, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                                "sample": smp.describe()}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        dist.destroy_process_group()
    return 0


def run_sweep(args):
    """Averaging-only sweep (P = 128): local, global and fused local+global GB/s."""
    import torch
    from paper_1903_05133_gb300 import configs
    from paper_1903_05133_gb300.hier_avg import (global_average_buffer, local_average_buffer,
                                                 local_global_average_buffer)
    sw = configs.AVERAGING_SWEEP
    pk, src = peaks()
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device="cuda")
    torch.manual_seed(0)
    for D in args.sweep_D or sw.D:
        w = torch.randn(sw.P, D, device="cuda")
        by = 8.0 * sw.P * D
        for op, S in [("global", sw.P)] + [(o, s) for s in sw.S for o in ("local", "local_global")]:
            fn = {"local": lambda: local_average_buffer(w, S),
                  "global": lambda: global_average_buffer(w),
                  "local_global": lambda: local_global_average_buffer(w, S)}[op]
            for _ in range(3):
                fn()
            ms = []
            for _ in range(max(5, args.steps // 5)):
                flush.zero_()
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record()
                fn()
                b.record()
                torch.cuda.synchronize()
                ms.append(a.elapsed_time(b))
            med = statistics.median(ms)
            gbs = by / (med / 1e3) / 1e9
            print(json.dumps({"P": sw.P, "D": D, "S": S, "op": op, "ms": round(med, 4),
                              "GBps": round(gbs, 1), "frac_hbm": round(gbs / pk["hbm_gbs"], 4),
                              "peak_source": src}), flush=True)
        del w
        torch.cuda.empty_cache()
    return 0


def main():
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
