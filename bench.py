#!/usr/bin/env python3
"""Benchmark of DARTree draft-tree construction on GB300.

One step = one full round of the hot path on one batch of synthetic input:
Algorithm 1 for depths 1..L (LM-head scoring with fused log-softmax/top-k,
frontier selection, correction-head update) followed by top-B pruning and
emission of the verification tree, launched through the C ABI
(dart_build_tree, one cached CUDA graph per round).

Prints ONE JSON line (rank 0).  `value` = node expansions per second over all
ranks (each rank builds its own replica rounds; no data-path collective).
Also reported: µs per round, the LM-head stream's HBM bandwidth, a roofline
object for the LM-head kernel, an end-to-end number through the host-buffer
entry point, clocks sampled during the timed region, and the CPU oracle timed
on a bounded sample of the same workload.

`--impl reference` times the fp64 CPU oracle (the reference arm of this
build) on the same workload and metric.
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

import numpy as np  # noqa: E402

METRIC = ("tree-construction µs/round and node expansions/s; LM-head HBM GB/s vs 8 TB/s")
UNIT = "node expansions/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="dart", choices=["dart", "reference"])
    ap.add_argument("--config", default="qwen3-8b")
    ap.add_argument("--cpu-seconds", type=float, default=15.0, help="oracle sample budget")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def allreduce_max(x, world, device=None):
    """Max of a float over all ranks (the timing rule: the job is as slow as
    its slowest rank).  No-op for a single process."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_step_per_rank, world, seconds_per_step):
    """Units of all ranks per second (weak scaling: every rank does the same
    amount of independent work)."""
    return units_per_step_per_rank * world / seconds_per_step


def measured_peak():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            j = json.load(f)
        return float(j["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_sha():
    h = hashlib.sha256()
    for f in ("dart_tc.cu", "dart_device.cuh"):
        with open(os.path.join(ROOT, "paper_2608_13524_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(workload):
    """DRAM bytes per LM-head launch from the committed ncu summary, if it was
    taken on the current kernel source."""
    p = os.path.join(ROOT, "profiles", "lmhead_traffic.json")
    try:
        with open(p) as f:
            j = json.load(f)
        e = j.get(workload)
        if e and e.get("source_sha") == kernel_source_sha():
            return float(e["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""

    Q = ("pci.bus_id,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.bus_id = bus_id
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                                          "-lms", "200"], stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.f.flush()
        rows = []
        with open(self.f.name) as fh:
            for line in fh:
                c = [x.strip() for x in line.split(",")]
                if len(c) < 9:
                    continue
                if self.bus_id and self.bus_id.lower() not in c[0].lower() and c[0].lower() not in self.bus_id.lower():
                    continue
                rows.append(c)
        os.unlink(self.f.name)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows)}


def cpu_baseline(cfg, x, budget_s):
    """The fp64 oracle, as it stands, on a bounded sample of the workload:
    node expansions (children of one prefix over the full vocabulary or over
    C_d + log-softmax + top-k, then the head update of one kept child) until
    the time budget is spent.  Returns expansions/s."""
    import oracle
    oracle.build()
    t0 = time.perf_counter()
    n = 0
    path = np.zeros(0, np.int32)
    while True:
        tok, lq, lse, _ = oracle.node_children(cfg, x["Wi"], x["Wo"], x["E"], x["Dlog"][0], x["h0"][0], path,
                                               cfg.k)
        if len(path) + 1 < cfg.L:
            oracle.head(cfg, x["Wi"], x["Wo"], x["E"], np.zeros(cfg.d), int(tok[0]))
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s or n >= 10000:
            break
    scope = "full-vocabulary" if cfg.cand_k == 0 else f"candidate-restricted (K={cfg.cand_k})"
    return dict(value=n / el, unit=UNIT, cores=oracle.num_threads(), kind="oracle",
                sample=f"{n} node expansions of {cfg.name} (V={cfg.V}, d={cfg.d}) at depth 1 "
                       f"({scope} fp64 scoring + one head update each), {el:.1f} s")


def run_reference(args, cfg):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from workloads import make_inputs
    x = make_inputs(cfg)
    budget = max(2.0, min(args.cpu_seconds, 60.0 / max(1, args.steps + args.warmup)))
    vals = []
    bl = None
    for i in range(args.warmup + args.steps):
        r = cpu_baseline(cfg, x, budget)
        if i >= args.warmup:
            vals.append(r["value"])
            bl = r
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name, "nseq": cfg.nseq, "V": cfg.V, "d": cfg.d, "L": cfg.L,
                       "W": cfg.W, "k": cfg.k, "B": cfg.B},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": bl["cores"], "kind": "oracle",
                             "sample": bl["sample"]},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.warmup < 3:
        args.warmup = 3
    from workloads import NAMED
    cfg = NAMED[args.config]
    if args.impl == "reference":
        run_reference(args, cfg)
        return

    import torch
    import torch.distributed as dist

    rank, world, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)

    from paper_2608_13524_gb300 import dart
    from workloads import make_inputs

    x = make_inputs(cfg, rank=rank)  # each replica builds its own sequences
    tb = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)
    tf = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    conv = tb if cfg.wdtype == "bf16" else tf
    Wi, Wo, E = conv(x["Wi"]), conv(x["Wo"]), conv(x["E"])
    D = tf(x["Dlog"])
    h0 = tf(x["h0"])
    stream = torch.cuda.current_stream(dev)
    eng = dart.Dart(cfg, Wi, Wo, E)
    h = eng.h
    launches = dart.dart_launches_per_round(h)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    # warm-up (also captures and instantiates the round's CUDA graph)
    for _ in range(args.warmup):
        eng.build_tree(D, h0, stream)
    rc = dart.dart_status_sync(h, stream)
    if rc != 0:
        raise RuntimeError(f"device status {rc} after warm-up")

    props = torch.cuda.get_device_properties(dev)
    bus = None
    try:
        bus = f"{props.pci_domain_id:08X}:{props.pci_bus_id:02X}:{props.pci_device_id:02X}.0"
    except Exception:
        pass
    clocks = ClockSampler(bus)
    clocks.start()
    time.sleep(0.3)

    # timed region: K rounds, graph launches, inputs resident in HBM.
    # Full vocabulary: E (V*d*2 bytes) is far larger than L2 and is streamed
    # once per depth, so rounds run back to back.  Candidate-restricted: the
    # bytes a round reads (head weights, K rows of E) fit in L2, so L2 is
    # flushed (a 512 MB write, untimed) before every timed round, as the
    # target model's verification pass would between two draft rounds.
    flush = torch.empty(128 * 1024 * 1024, dtype=torch.float32, device=dev) if cfg.cand_k > 0 else None
    barrier()
    if flush is None:
        ev0 = torch.cuda.Event(enable_timing=True)
        ev1 = torch.cuda.Event(enable_timing=True)
        ev0.record(stream)
        for _ in range(args.steps):
            eng.build_tree(D, h0, stream)
        ev1.record(stream)
        barrier()
        ms_local = ev0.elapsed_time(ev1) / args.steps
    else:
        evs = []
        for i in range(args.steps):
            with torch.cuda.stream(stream):
                flush.fill_(float(i))
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            eng.build_tree(D, h0, stream)
            b.record(stream)
            evs.append((a, b))
        barrier()
        ms_local = sum(a.elapsed_time(b) for a, b in evs) / args.steps
    ms = allreduce_max(ms_local, world, dev)
    clk = clocks.stop()
    rc = dart.dart_status_sync(h, stream)
    if rc != 0:
        raise RuntimeError(f"device status {rc} after timed region")

    # LM-head kernel duration: the same rounds with CUDA events around every
    # LM-head launch on the launching stream (direct launches, no graph).
    dart.dart_set_profiling(h, True)
    for _ in range(2):
        eng.build_tree(D, h0, stream)
    dart.dart_profile_read(h)
    barrier()
    pe0 = torch.cuda.Event(enable_timing=True)
    pe1 = torch.cuda.Event(enable_timing=True)
    pe0.record(stream)
    for _ in range(args.steps):
        eng.build_tree(D, h0, stream)
    pe1.record(stream)
    barrier()
    prof_ms_round = pe0.elapsed_time(pe1) / args.steps
    kinds = dart.dart_profile_read_kinds(h)
    dart.dart_set_profiling(h, False)
    # roofline kernel: the LM-head stream, or with candidate-restricted
    # scoring the largest remaining HBM stream, the W_i GEMM (2*d*d weights)
    rl_kind = "lmhead" if cfg.cand_k == 0 else "gemm_wi"
    k1_ms, k1_n = kinds[rl_kind]
    k1_avg_s = k1_ms / 1e3 / max(1, k1_n)
    breakdown = {k: {"us_per_round": v[0] * 1e3 / args.steps, "launches_per_round": v[1] / args.steps,
                     "us_per_launch": v[0] * 1e3 / max(1, v[1])} for k, v in kinds.items() if v[1]}

    exp_round = cfg.expansions_per_round()
    value = whole_job_rate(exp_round, world, ms / 1e3)
    bytes_launch = cfg.lmhead_bytes_per_depth() if cfg.cand_k == 0 else 2 * cfg.d * cfg.d * cfg.bpe
    lm_bytes_round = cfg.L * cfg.V * cfg.d * cfg.bpe if cfg.cand_k == 0 else None
    peak, peak_kind = measured_peak()
    achieved = bytes_launch / k1_avg_s / 1e9
    traffic = recorded_traffic(cfg.name)

    # end to end through the host-buffer entry point (H2D of the inputs and
    # D2H of the emitted tree inside the timed region)
    e2e = None
    if not args.no_e2e:
        Dh = torch.from_numpy(x["Dlog"]).pin_memory()
        hh = torch.from_numpy(x["h0"]).pin_memory()
        ht, hout = dart.alloc_tree_out(cfg, pin=True)
        for _ in range(2):
            dart.dart_build_tree_host(h, Dh, hh, hout, stream)
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            dart.dart_build_tree_host(h, Dh, hh, hout, stream)
        barrier()
        e2e_s = allreduce_max((time.perf_counter() - t0) / args.steps, world, dev)
        h2d = Dh.numel() * 4 + hh.numel() * 4
        d2h = sum(v.numel() * v.element_size() for v in ht.values())
        e2e = {"value": whole_job_rate(exp_round, world, e2e_s), "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_s * 1e3}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(cfg, x, args.cpu_seconds)

    eng.close()
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16" if cfg.wdtype == "bf16" else "f32",
            "data": "synthetic",
            "config": {"workload": cfg.name, "nseq": cfg.nseq, "V": cfg.V, "d": cfg.d, "L": cfg.L,
                       "W": cfg.W, "k": cfg.k, "B": cfg.B, "K": cfg.cand_k if cfg.cand_k else "full vocabulary",
                       "beta": cfg.beta, "T": cfg.temperature,
                       "parallelism": f"replicas x{world}",
                       "l2": ("inputs larger than L2: E (%.2f GB) streamed once per depth" %
                              (cfg.V * cfg.d * cfg.bpe / 1e9)) if cfg.cand_k == 0 else
                             ("L2 flushed (512 MB write, untimed) before every timed round; the round's "
                              "head weights (%.0f MB) would fit in L2" % (3 * cfg.d * cfg.d * cfg.bpe / 1e6))},
            "us_per_round": ms * 1e3,
            "lmhead_gbs": lm_bytes_round / (ms / 1e3) / 1e9 if lm_bytes_round else None,
            "lmhead_frac_of_8tbs": lm_bytes_round / (ms / 1e3) / 1e9 / NOMINAL_HBM_GBS if lm_bytes_round else None,
            "roofline": {"kernel": "lmhead_tc_kernel" if cfg.cand_k == 0 else "gemm_tc_kernel (W_i)",
                         "bound": "hbm", "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "GB/s", "frac": achieved / peak,
                         "traffic": traffic, "bytes_per_launch": bytes_launch,
                         "avg_launch_us": k1_avg_s * 1e6, "launches": k1_n,
                         "profiled_us_per_round": prof_ms_round * 1e3},
            "kernel_breakdown": breakdown,
            "gpu_launches": launches * args.steps,
            "clocks": clk,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
