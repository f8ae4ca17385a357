#!/usr/bin/env python3
"""Throughput of the Hier-AVG hot path on GB300.

One bench "step" is one global round of Algorithm 1 (Sec. 3.1): K2 x (K1 local
SGD steps of all P learners + a local average) + the global average, on
synthetic Gaussian-mixture data already resident in HBM.  The metric is
learner-samples per second (P * B * K1 * K2 per round).

  python bench.py [--gpus N --steps K --warmup W] [--workload mlp512|mlp2048|mlp4096|softmax]
  python bench.py --impl reference ...   # the CPU oracle on a bounded sample
  python bench.py --sweep                # averaging-only sweep (P = 128), GB/s table

Under torchrun (N > 1) every rank runs an independent replica on its own GPU
(the learners of one replica never leave their GPU), timing is max over ranks
and ``value`` is the sum over replicas ("scaling": "weak").
"""
from __future__ import annotations

import argparse
import hashlib
import json
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
DOM_SAMPLE = 7   # time 1 in 7 launches of the dominant kernel (coprime with the layer counts)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="mlp512")
    ap.add_argument("--sweep", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
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


def ncu_traffic(kind: str, workload: str):
    """DRAM bytes per launch of a kernel from a committed ncu summary, if the
    kernel source has not changed since it was captured."""
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
    return e.get("dram_bytes_per_launch")


# ----------------------------------------------------------------------------- oracle
def oracle_block_time(w, X, y, layers, n_blocks: int = 1):
    """Time the CPU oracle on one local block (K1 local steps of every learner +
    one local average) per call; returns (seconds per block, samples per block)."""
    import numpy as np
    import oracle
    mode = "fp32" if w.precision == "fp32" else "bf16"
    params = []
    for Wl, bl in layers:
        params += [np.broadcast_to(Wl.numpy(), (w.P,) + tuple(Wl.shape)).copy(),
                   np.broadcast_to(bl.numpy(), (w.P,) + tuple(bl.shape)).copy()]
    prob = oracle.MLPProblem(X.float().numpy(), y.numpy().astype(np.int64), w.B, len(w.dims) - 1, mode)
    o = oracle.HierAvgOracle(w.P, w.S, w.K1, w.K2, w.lr, prob, params, mode)
    times = []
    for _ in range(n_blocks):
        t0 = time.perf_counter()
        for _k in range(w.K1):
            o.step()
        o.local_average()
        times.append(time.perf_counter() - t0)
    return times, w.P * w.B * w.K1


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def run_reference(args):
    ws, rank, _ = dist_env()
    if rank != 0:
        return 0
    from paper_1903_05133_gb300 import configs
    from paper_1903_05133_gb300.inputs import initial_layers, learner_data
    w = configs.SHORT[args.workload]
    X, y = learner_data(w)
    layers = initial_layers(w)
    times, samples = oracle_block_time(w, X, y, layers, args.warmup + args.steps)
    timed = times[args.warmup:]
    T = sum(timed)
    value = samples * len(timed) / T
    sample = (f"one local block per step: {w.K1} local SGD steps of all {w.P} learners + one local "
              f"average ({samples} learner-samples, 1/{w.K2} of a round; the global average is "
              f"not in the sample)")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * T / len(timed),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16-operands/f64-acc",
            "data": "synthetic", "config": {"workload": w.name, "P": w.P, "S": w.S, "K1": w.K1,
                                            "K2": w.K2, "B": w.B, "dims": list(w.dims)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- ours
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
    dom = max(main_kinds, key=lambda k: prof[k][0])

    props = torch.cuda.get_device_properties(dev)
    uuid = str(getattr(props, "uuid", "") or "")
    sampler = ClockSampler()
    time.sleep(0.05)
    # one launch in DOM_SAMPLE of the dominant kernel is timed (events separate it from
    # its neighbours; timing every launch cost ~9 % of the round at 3072-512-10)
    ha.profile([dom])
    ha.profile_every(DOM_SAMPLE)
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
    dom_ms, dom_n, dom_bytes = dom_live
    achieved = dom_bytes / (dom_ms / 1e3) / 1e9 if dom_ms > 0 else None
    kernels = {}
    for k in kinds:
        ms, n, by = prof[k]
        if n:
            kernels[k] = {"launches": n, "total_ms": round(ms, 4), "avg_us": round(1e3 * ms / n, 2),
                          "share": round(ms / max(1e-9, sum(v[0] for v in prof.values())), 4),
                          "GBps": round(by / (ms / 1e3) / 1e9, 1) if ms > 0 else None}
    avg_ms = prof["local_avg"][0] + prof["global_avg"][0]
    avg_by = prof["local_avg"][2] + prof["global_avg"][2]
    # per-launch DRAM bytes scale with P: a run with fewer learners has no captured figure
    traffic = ncu_traffic(dom, w.name) if not args.P else None
    roofline = {"kernel": dom, "bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "frac": (achieved / pk["hbm_gbs"]) if achieved else None,
                "peak_source": pk_src,
                "traffic": traffic,
                "algorithmic_bytes_per_launch": dom_bytes / max(1, dom_n),
                "avg_launch_us": 1e3 * dom_ms / max(1, dom_n),
                "timing": f"CUDA events around every {DOM_SAMPLE}th launch of this kernel inside the timed rounds",
                "launches_timed": dom_n}

    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": 1000 * T / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.precision,
            "data": "synthetic (seeded Gaussian mixture, CIFAR-10 / ImageNet shaped)",
            "config": {"workload": w.name, "P": w.P, "S": w.S, "K1": w.K1, "K2": w.K2, "B": w.B,
                       "dims": list(w.dims), "lr": w.lr, "N": w.N,
                       "parallelism": f"{w.P} simulated learners per GPU" + (f" x {ws} replicas" if ws > 1 else ""),
                       "l2": f"flushed between timed rounds ({L2_FLUSH_BYTES >> 20} MB write, untimed)",
                       "master": "fp32", "gemm_operands": w.precision},
            "roofline": roofline,
            "averaging": {"GBps": avg_by / (avg_ms / 1e3) / 1e9 if avg_ms > 0 else None,
                          "frac_of_measured_hbm": (avg_by / (avg_ms / 1e3) / 1e9 / pk["hbm_gbs"]) if avg_ms > 0 else None,
                          "frac_of_8TBps": (avg_by / (avg_ms / 1e3) / 8e12) if avg_ms > 0 else None},
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
        t0 = time.perf_counter()
        for _ in range(args.steps):
            ha.round_host(Xh, yh, loss)
        torch.cuda.synchronize()
        Te = job_seconds(time.perf_counter() - t0, ws, dev)
        rows = w.B * w.K1 * w.K2
        es = 2 if w.precision == "bf16" else 4
        line["e2e"] = {"value": replica_throughput(ws, per_round, args.steps, Te), "unit": UNIT,
                       "h2d_bytes_per_step": w.P * rows * (w.dims[0] * es + 4),
                       "d2h_bytes_per_step": w.P * 4,
                       "api": "hier_avg_round_host (pinned host X, y; loss read back)"}

    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        Xc, yc = X.cpu(), y.cpu()
        lc = [(Wl.cpu(), bl.cpu()) for Wl, bl in layers]
        times, samples = oracle_block_time(w, Xc, yc, lc, 1)
        line["cpu_baseline"] = {"value": samples / times[0], "unit": UNIT, "cores": cpu_cores(),
                                "kind": "oracle",
                                "sample": f"one local block: {w.K1} local steps of all {w.P} learners "
                                          f"+ one local average ({samples} learner-samples), numpy "
                                          f"(float64 BLAS products, multi-threaded BLAS)"}
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
    for D in sw.D:
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
