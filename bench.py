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


def code_sha(files):
    """Hash of CUDA sources with comments and blank space removed: a capture
    stays valid across comment-only edits and is void after any code change."""
    import re
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2608_13524_gb300", "csrc", f)) as fh:
            src = fh.read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


def kernel_source_sha():
    return code_sha(("dart_tc.cu", "dart_device.cuh"))


def split_head(cfg):
    """True when the library splits the first head layer (bf16 weights):
    each depth streams W_i[:, 0:d] (2 d^2 bytes) instead of all of W_i."""
    return cfg.wdtype == "bf16" and cfg.head_split != 2


def wi_bytes_per_depth(cfg):
    return (1 if split_head(cfg) else 2) * cfg.d * cfg.d * cfg.bpe


def kept_head_weights(cfg):
    """(W_i kept, W_o kept): the head weights the library loads evict-last
    so that they stay in L2 across the depths of a round.  Mirrors its plan:
    candidate-restricted scoring, <= 16 children, the largest of {both, W_i
    (its first half with the split first layer), W_o} within 72 MiB (bf16
    weights)."""
    if cfg.cand_k == 0 or cfg.wdtype != "bf16" or cfg.nseq * cfg.W > 16:
        return False, False
    cap = 72 << 20
    wi, wo = wi_bytes_per_depth(cfg), 2 * cfg.d * cfg.d
    if wi + wo <= cap:
        return True, True
    return wi <= cap, wi > cap and wo <= cap


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


class L2Flush:
    """Untimed L2 flush between timed calls: write a 512 MB buffer (four
    times L2), then read another 512 MB buffer, so the write-back of the dirty
    flush lines happens here and not inside the next timed kernel; the timed
    call starts from an L2 holding only unrelated clean lines."""

    def __init__(self, dev):
        import torch
        self.torch = torch
        self.w = torch.empty(128 * 1024 * 1024, dtype=torch.float32, device=dev)
        self.r = torch.ones(128 * 1024 * 1024, dtype=torch.float32, device=dev)
        self.sink = torch.empty((), dtype=torch.float32, device=dev)

    def __call__(self, stream, i):
        with self.torch.cuda.stream(stream):
            self.w.fill_(float(i))
            self.torch.sum(self.r, dim=0, out=self.sink)


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


# ------------------------------------------------------------------ tree attention
# (the verification consumer of the emitted tree, Sec. 3.3: one attention
# layer over [context ; tree] with the ancestor mask and the tree positions)

ATTN_METRIC = "tree-attention verification layer: tree tokens/s (µs per call)"
ATTN_UNIT = "tree tokens/s"


def measured_tflops():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            return float(json.load(f)["bf16_tflops"]), "measured (bf16 burst)"
    except Exception:
        return 1900.0, "fallback (bf16 burst)"


def attn_source_sha():
    return code_sha(("dart_attn.cu", "dart_device.cuh"))


def attn_recorded_traffic(workload):
    p = os.path.join(ROOT, "profiles", "attn_traffic.json")
    try:
        with open(p) as f:
            e = json.load(f).get(workload)
        if e and e.get("source_sha") == attn_source_sha():
            return float(e["dram_bytes_per_launch"])
    except Exception:
        pass
    return None


def attn_flops(acfg, x):
    """Algorithmic FLOPs of one call: 2 * dh multiply-adds for q.k and for
    p*v per (tree row, query head, visible key); visible keys = the context
    plus the row's root-to-node path (its depth)."""
    vis = 0
    for s in range(acfg.nseq):
        n = int(x["n_nodes"][s])
        vis += n * acfg.C + int(x["depths"][s][:n].sum())
    return 4.0 * acfg.dh * acfg.Hq * vis


def attn_cpu_baseline(acfg, x, budget_s):
    """The fp64 oracle, as it stands, on a bounded sample: tree rows (all
    query heads each) of sequence 0 until the budget is spent."""
    from oracle import tree_attn as ta
    from workloads import bf16_bits_to_f32
    f = lambda a: bf16_bits_to_f32(a).astype(np.float64)
    q, kt, vt, kc, vc = f(x["q"]), f(x["k_tree"]), f(x["v_tree"]), f(x["k_ctx"]), f(x["v_ctx"])
    t0 = time.perf_counter()
    rows = 0
    n = int(x["n_nodes"][0])
    while True:
        ta.tree_attention(q, kt, vt, kc, vc, x["parents"], x["depths"], x["n_nodes"], acfg.offset,
                          acfg.rope_theta, acfg.scale, rows=[(0, rows % n)])
        rows += 1
        el = time.perf_counter() - t0
        if el >= budget_s or rows >= 100000:
            break
    return dict(value=rows / el, unit=ATTN_UNIT, cores=blas_threads(), kind="oracle",
                sample=f"{rows} tree rows x {acfg.Hq} query heads of {acfg.name} (C={acfg.C}, dh={acfg.dh}), "
                       f"fp64 path-walk attention, {el:.1f} s")


def blas_threads():
    """Threads numpy's BLAS may use (the oracle's matrix-vector products)."""
    try:
        from threadpoolctl import threadpool_info
        n = [p["num_threads"] for p in threadpool_info() if p.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return os.cpu_count() or 1


def attn_config_json(acfg, world, x):
    return {"workload": acfg.name, "nseq": acfg.nseq, "B": acfg.B, "C": acfg.C, "Hq": acfg.Hq, "Hkv": acfg.Hkv,
            "dh": acfg.dh, "rope_theta": acfg.rope_theta, "tree": f"random prefix tree, L={acfg.L}, W={acfg.W}",
            "n_nodes": [int(v) for v in x["n_nodes"]], "parallelism": f"replicas x{world}",
            "l2": "L2 flushed before every timed call (untimed 512 MB write, then a 512 MB read that takes the "
                  "write-back): the KV cache fits in L2"}


def run_verify_reference(args, acfg):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    from workloads import make_attn_inputs
    x = make_attn_inputs(acfg)
    budget = max(2.0, min(args.cpu_seconds, 60.0 / max(1, args.steps + args.warmup)))
    vals, bl = [], None
    for i in range(args.warmup + args.steps):
        r = attn_cpu_baseline(acfg, x, budget)
        if i >= args.warmup:
            vals.append(r["value"])
            bl = r
    v = statistics.median(vals)
    line = {"impl": "reference", "metric": ATTN_METRIC, "value": v, "unit": ATTN_UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": attn_config_json(acfg, world, x),
            "cpu_baseline": {"value": v, "unit": ATTN_UNIT, "cores": bl["cores"], "kind": "oracle",
                             "sample": bl["sample"]},
            "e2e": {"value": v, "unit": ATTN_UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_verify(args, acfg):
    import torch
    import torch.distributed as dist

    rank, world, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    from paper_2608_13524_gb300 import dart
    from workloads import make_attn_inputs

    x = make_attn_inputs(acfg)
    bf = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)
    q, kt, vt = bf(x["q"]), bf(x["k_tree"]), bf(x["v_tree"])
    kc = bf(x["k_ctx"]) if acfg.C > 0 else None
    vc = bf(x["v_ctx"]) if acfg.C > 0 else None
    par = torch.from_numpy(x["parents"]).to(dev)
    nn = torch.from_numpy(x["n_nodes"]).to(dev)
    dep = torch.from_numpy(x["depths"]).to(dev)
    pos = torch.where(dep > 0, dep + acfg.offset, torch.full_like(dep, -1)).to(torch.int32)
    mask = torch.empty((acfg.nseq, acfg.B, (acfg.B + 63) // 64), dtype=torch.int64, device=dev)
    stream = torch.cuda.current_stream(dev)
    dart.dart_ancestor_mask(par, nn, mask, stream)
    att = dart.TreeAttention(acfg.nseq, acfg.B, acfg.C, acfg.Hq, acfg.Hkv, acfg.dh, acfg.rope_theta, acfg.scale)
    status = torch.zeros(4, dtype=torch.int32, device=dev)
    call = lambda: att(q, kt, vt, kc, vc, pos, mask, nn, status, stream)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for _ in range(args.warmup):
        call()
    barrier()
    if int(status[0].item()) != 0:
        raise RuntimeError("device status after warm-up")
    props = torch.cuda.get_device_properties(dev)
    bus = None
    try:
        bus = f"{props.pci_domain_id:08X}:{props.pci_bus_id:02X}:{props.pci_device_id:02X}.0"
    except Exception:
        pass
    clocks = ClockSampler(bus)
    clocks.start()
    time.sleep(0.3)
    # the KV cache (and everything else a call reads) fits in L2: flush it
    # (untimed) before every timed call
    flush = L2Flush(dev)
    barrier()
    evs = []
    for i in range(args.steps):
        flush(stream, i)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        call()
        b.record(stream)
        evs.append((a, b))
    barrier()
    ms = allreduce_max(sum(a.elapsed_time(b) for a, b in evs) / args.steps, world, dev)
    clk = clocks.stop()
    if int(status[0].item()) != 0:
        raise RuntimeError("device status after the timed region")
    # attention kernel duration (events around its launch, same flushed calls)
    rope_ms, attn_ms = [], []
    for i in range(args.steps):
        flush(stream, i)
        r, k = att.timed(q, kt, vt, kc, vc, pos, mask, nn, status, stream)
        rope_ms.append(r)
        attn_ms.append(k)
    k_s = statistics.mean(attn_ms) / 1e3
    flops = attn_flops(acfg, x)
    peak, peak_kind = measured_tflops()
    achieved = flops / k_s / 1e12
    tokens = int(sum(int(v) for v in x["n_nodes"]))
    value = whole_job_rate(tokens, world, ms / 1e3)

    e2e = None
    if not args.no_e2e:
        hq, hkt, hvt = (torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).pin_memory()
                        for a in (x["q"], x["k_tree"], x["v_tree"]))
        hpos = pos.cpu().pin_memory()
        hmask = mask.cpu().pin_memory()
        hnn = nn.cpu().pin_memory()
        hout = torch.empty(att.out.shape, dtype=torch.float32).pin_memory()
        dq, dkt, dvt = torch.empty_like(q), torch.empty_like(kt), torch.empty_like(vt)

        def e2e_call():
            with torch.cuda.stream(stream):
                dq.view(torch.int16).copy_(hq, non_blocking=True)
                dkt.view(torch.int16).copy_(hkt, non_blocking=True)
                dvt.view(torch.int16).copy_(hvt, non_blocking=True)
                pos.copy_(hpos, non_blocking=True)
                mask.copy_(hmask, non_blocking=True)
                nn.copy_(hnn, non_blocking=True)
            att(dq, dkt, dvt, kc, vc, pos, mask, nn, status, stream)
            with torch.cuda.stream(stream):
                hout.copy_(att.out, non_blocking=True)

        for _ in range(2):
            e2e_call()
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            e2e_call()
        barrier()
        e2e_s = allreduce_max((time.perf_counter() - t0) / args.steps, world, dev)
        h2d = sum(v.numel() * v.element_size() for v in (hq, hkt, hvt, hpos, hmask, hnn))
        e2e = {"value": whole_job_rate(tokens, world, e2e_s), "unit": ATTN_UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": hout.numel() * 4, "ms_per_step": e2e_s * 1e3,
               "note": "tree q/k/v, positions, mask and n_nodes copied in from pinned host memory and the "
                       "output copied out every call; the context KV cache stays resident"}
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = attn_cpu_baseline(acfg, x, args.cpu_seconds)
    if rank == 0:
        line = {
            "metric": ATTN_METRIC, "value": value, "unit": ATTN_UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": attn_config_json(acfg, world, x),
            "us_per_call": ms * 1e3,
            "roofline": {"kernel": "tree_attn_kernel", "bound": "tensor", "achieved": achieved, "peak": peak,
                         "peak_kind": peak_kind, "unit": "TFLOP/s", "frac": achieved / peak,
                         "traffic": attn_recorded_traffic(acfg.name), "flops_per_launch": flops,
                         "avg_launch_us": k_s * 1e6, "rope_prepass_us": statistics.mean(rope_ms) * 1e3},
            "gpu_launches": 2 * args.steps,
            "clocks": clk,
            "e2e": e2e,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


# ------------------------------------------------------- extra measurement modes

def gpu_setup():
    import torch
    import torch.distributed as dist
    rank, world, local = dist_env()
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else 0)
    torch.cuda.set_device(dev)
    return rank, world, dev


def device_inputs(cfg, x, dev):
    import torch
    tb = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev).view(torch.bfloat16)
    tf = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    conv = tb if cfg.wdtype == "bf16" else tf
    return conv(x["Wi"]), conv(x["Wo"]), conv(x["E"]), tf(x["Dlog"]), tf(x["h0"])


def clock_sampler(dev):
    import torch
    props = torch.cuda.get_device_properties(dev)
    bus = None
    try:
        bus = f"{props.pci_domain_id:08X}:{props.pci_bus_id:02X}:{props.pci_device_id:02X}.0"
    except Exception:
        pass
    return ClockSampler(bus)


def time_rounds(build, steps, stream, barrier):
    """Average device ms of `steps` back-to-back rounds (CUDA events on the
    launching stream; the caller warmed up)."""
    import torch
    barrier()
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    for _ in range(steps):
        build()
    b.record(stream)
    barrier()
    return a.elapsed_time(b) / steps


def profile_round(dart, h, build, steps, barrier):
    """Per-kind device time and launch count of `steps` rounds (events around
    every launch, direct launches), averaged per round."""
    dart.dart_set_profiling(h, True)
    build()
    dart.dart_profile_read_kinds(h)
    barrier()
    for _ in range(steps):
        build()
    barrier()
    kinds = dart.dart_profile_read_kinds(h)
    dart.dart_set_profiling(h, False)
    return {k: (v[0] / steps, v[1] / steps) for k, v in kinds.items() if v[1]}


def run_table2(args, base):
    """Construction-only latency of the tree constructions of Table 2 and of
    DARTree (fixed) on the same synthetic inputs: DARTree (the workload's W,
    k, B, pruned), DARTree (fixed) (W = k = B / L, no pruning), Domino-chain +
    DDTree and sequential correction with heap (both with the workload's B)."""
    import torch
    from paper_2608_13524_gb300 import dart
    from workloads import make_inputs

    rank, world, dev = gpu_setup()
    cfg = base.replace(variants=3)
    wf = max(1, cfg.B // cfg.L)
    fixed = base.replace(name=base.name + "-fixed", W=wf, k=wf, B=wf * cfg.L)
    x = make_inputs(cfg, rank=rank)
    Wi, Wo, E, D, h0 = device_inputs(cfg, x, dev)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)

    eng = dart.Dart(cfg, Wi, Wo, E)
    engf = dart.Dart(fixed, Wi, Wo, E)
    cons = [("dartree", eng, lambda: eng.build_tree(D, h0, stream), cfg),
            ("dartree_fixed", engf, lambda: engf.build_tree_fixed(D, h0, stream), fixed),
            ("chain_ddtree", eng, lambda: eng.build_chain_ddtree(D, h0, stream), cfg),
            ("seq_heap", eng, lambda: eng.build_seq_heap(D, h0, stream), cfg)]
    for _, e, build, _ in cons:
        for _ in range(args.warmup):
            build()
        if dart.dart_status_sync(e.h, stream) != 0:
            raise RuntimeError("device status after warm-up")
    clocks = clock_sampler(dev)
    clocks.start()
    time.sleep(0.3)
    ms = {name: allreduce_max(time_rounds(build, args.steps, stream, barrier), world, dev)
          for name, _, build, _ in cons}
    clk = clocks.stop()
    peak, peak_kind = measured_peak()
    out = {}
    launches = 0
    for name, e, build, c in cons:
        kinds = profile_round(dart, e.h, build, 2, barrier)  # up to ~2300 launches per round: 2 fit the event pool
        lm_ms, lm_n = kinds.get("lmhead", (0.0, 0))
        n_launch = sum(v[1] for v in kinds.values())
        launches += n_launch * args.steps
        emitted = tree_to_counts(e.out_t)
        out[name] = {"us_per_round": ms[name] * 1e3, "vs_dartree": ms[name] / ms["dartree"],
                     "lmhead_launches_per_round": lm_n, "launches_per_round": n_launch,
                     "lmhead_us_per_launch": lm_ms * 1e3 / max(lm_n, 1e-9),
                     "lmhead_hbm_frac": (c.V * c.d * c.bpe + c.V * 4) / (lm_ms / 1e3 / max(lm_n, 1e-9)) / 1e9 / peak
                     if lm_n else None,
                     "W": c.W, "k": c.k, "B": c.B, "nodes_emitted": emitted,
                     "kernel_us_per_round": {k: v[0] * 1e3 for k, v in kinds.items()}}
    if dart.dart_status_sync(eng.h, stream) != 0 or dart.dart_status_sync(engf.h, stream) != 0:
        raise RuntimeError("device status after the timed region")
    eng.close()
    engf.close()
    if rank == 0:
        line = {"metric": "tree-construction µs/round, the constructions of Table 2 on one input",
                "value": ms["dartree"] * 1e3, "unit": "µs/round", "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": sum(ms.values()), "higher_is_better": False,
                "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if cfg.wdtype == "bf16" else "f32",
                "data": "synthetic",
                "config": {"workload": base.name, "nseq": cfg.nseq, "V": cfg.V, "d": cfg.d, "L": cfg.L,
                           "beta": cfg.beta, "T": cfg.temperature, "parallelism": f"replicas x{world}",
                           "l2": "inputs larger than L2: E streamed by every LM-head pass"},
                "constructions": out, "gpu_launches": int(launches), "clocks": clk, "peak_hbm_gbs": peak,
                "peak_kind": peak_kind,
                "paper_context": "Table 2 (Qwen3-4B, GSM8K, B = 64, RTX 6000 Ada, whole rounds incl. drafting "
                                 "and verification): DARTree 28.494 ms, Domino-chain + DDTree 28.285 ms, "
                                 "Seq. correction w. heap 62.703 ms",
                "e2e": None, "cpu_baseline": None}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def tree_to_counts(out_t):
    return [int(v) for v in out_t["n_nodes"].cpu().tolist()]


def run_sweep(args):
    """The width / budget sweep at the Qwen3-4B shape (Sec. 5.3): every
    (W, B) point, µs per round, the LM-head kernel's time per launch and its
    fraction of the measured HBM copy peak, the round's LM-head bytes over
    the round time against 8 TB/s."""
    import torch
    from paper_2608_13524_gb300 import dart
    from workloads import make_inputs, sweep_configs

    rank, world, dev = gpu_setup()
    pts = sweep_configs()
    x = make_inputs(pts[0], rank=rank)
    Wi, Wo, E, D, h0 = device_inputs(pts[0], x, dev)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if world > 1:
            torch.distributed.barrier()
        torch.cuda.synchronize(dev)

    peak, peak_kind = measured_peak()
    clocks = clock_sampler(dev)
    clocks.start()
    time.sleep(0.3)
    rows, launches, total_exp, total_ms = [], 0, 0, 0.0
    for cfg in pts:
        eng = dart.Dart(cfg, Wi, Wo, E)
        build = lambda: eng.build_tree(D, h0, stream)
        for _ in range(args.warmup):
            build()
        ms = allreduce_max(time_rounds(build, args.steps, stream, barrier), world, dev)
        kinds = profile_round(dart, eng.h, build, max(2, args.steps // 4), barrier)
        if dart.dart_status_sync(eng.h, stream) != 0:
            raise RuntimeError(f"device status after {cfg.name}")
        lm_ms, lm_n = kinds["lmhead"]
        lm_s = lm_ms / 1e3 / lm_n
        launches += dart.dart_launches_per_round(eng.h) * args.steps
        exp = cfg.expansions_per_round() * world
        total_exp += exp
        total_ms += ms
        rows.append({"W": cfg.W, "B": cfg.B, "us_per_round": ms * 1e3, "node_expansions_per_s": exp / (ms / 1e3),
                     "lmhead_us_per_launch": lm_s * 1e6,
                     "lmhead_hbm_frac": cfg.lmhead_bytes_per_depth() / lm_s / 1e9 / peak,
                     "round_lmhead_frac_of_8tbs": cfg.L * cfg.V * cfg.d * cfg.bpe / (ms / 1e3) / 1e9 / NOMINAL_HBM_GBS,
                     "nodes_emitted": min(cfg.B, sum(cfg.caps()[1:]))})
        eng.close()
    clk = clocks.stop()
    if rank == 0:
        line = {"metric": "tree-construction µs/round across the width / budget sweep", "value": total_exp / (total_ms / 1e3),
                "unit": "node expansions/s (all points)", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
                "ms_per_step": total_ms / len(pts), "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
                "dtype": "bf16", "data": "synthetic",
                "config": {"workload": "sweep (Qwen3-4B shape)", "V": pts[0].V, "d": pts[0].d, "L": pts[0].L,
                           "W": [8, 16, 32, 64], "k": "= W", "B": [32, 128, 512, 1024], "beta": pts[0].beta,
                           "T": pts[0].temperature, "parallelism": f"replicas x{world}",
                           "l2": "inputs larger than L2: E (0.78 GB) streamed once per depth"},
                "sweep": rows, "peak_hbm_gbs": peak, "peak_kind": peak_kind, "gpu_launches": int(launches),
                "clocks": clk, "e2e": None, "cpu_baseline": None}
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def ensure_ranks(args):
    """--gpus N: under torchrun WORLD_SIZE must be N; without it, N > 1
    relaunches this command as N local ranks (one per GPU) and returns the
    launcher's exit status."""
    world = os.environ.get("WORLD_SIZE")
    if world is not None:
        if int(world) != args.gpus:
            sys.stderr.write(f"bench.py: --gpus {args.gpus} but WORLD_SIZE={world}\n")
            return 2
        return None
    if args.gpus <= 1:
        return None
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        port = sk.getsockname()[1]
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args.gpus}",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__)] + sys.argv[1:]
    return subprocess.run(cmd).returncode


def main():
    args = parse()
    if args.warmup < 3:
        args.warmup = 3
    rc = ensure_ranks(args)
    if rc is not None:
        sys.exit(rc)
    from workloads import ATTN_NAMED, NAMED
    if args.config in ATTN_NAMED:
        acfg = ATTN_NAMED[args.config]
        if args.impl == "reference":
            run_verify_reference(args, acfg)
        else:
            run_verify(args, acfg)
        return
    if args.config == "sweep" and args.impl != "reference":
        run_sweep(args)
        return
    if args.config.startswith("table2-") and args.impl != "reference":
        run_table2(args, NAMED[args.config[len("table2-"):]])
        return
    cfg = NAMED[args.config if args.config in NAMED else args.config.split("table2-")[-1]] \
        if args.config != "sweep" else NAMED["sweep-W16-B128"]
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
    # flushed (L2Flush, untimed) before every timed round, as the target
    # model's verification pass would between two draft rounds.
    flush = L2Flush(dev) if cfg.cand_k > 0 else None
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
            flush(stream, i)
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
    # scoring the head GEMM whose weights stream from HBM at every depth (W_i
    # or, with the split first layer, its first half W_i[:, 0:d], else W_o);
    # when both stay in L2 the W_i GEMM with its weights counted once per
    # round (the HBM reads it needs)
    wi_kept, wo_kept = kept_head_weights(cfg)
    if kinds.get("round_f32", (0.0, 0))[1] > 0:
        # the fused small-problem round: one launch per round reads E and the
        # drafter rows once per depth and the head weights once per head update
        rl_kind, rl_name = "round_f32", "fused fp32 round kernel (whole round)"
        bytes_launch = cfg.L * cfg.lmhead_bytes_per_depth() + (cfg.L - 1) * 3 * cfg.d * cfg.d * cfg.bpe
        rl_note = "one launch per round; latency-bound (cluster or grid barriers between steps), its bytes fit in L2"
    elif cfg.cand_k == 0:
        rl_kind, rl_name, bytes_launch, rl_note = "lmhead", "lmhead_tc_kernel", cfg.lmhead_bytes_per_depth(), None
    elif not wi_kept:
        rl_kind, rl_name, bytes_launch, rl_note = "gemm_wi", "gemm_tc_kernel (W_i)", wi_bytes_per_depth(cfg), None
    elif not wo_kept:
        rl_kind, rl_name, bytes_launch, rl_note = ("gemm_wo", "gemm_tc_kernel (W_o)", cfg.d * cfg.d * cfg.bpe,
                                                   "W_i stays in L2 across depths; W_o streams from HBM")
    else:
        rl_kind, rl_name = "gemm_wi", "gemm_tc_kernel (W_i)"
        bytes_launch = wi_bytes_per_depth(cfg) / max(1, cfg.L - 1)
        rl_note = "W_i and W_o stay in L2 across depths: W_i bytes counted once per round"
    k1_ms, k1_n = kinds[rl_kind]
    k1_avg_s = k1_ms / 1e3 / max(1, k1_n)
    breakdown = {k: {"us_per_round": v[0] * 1e3 / args.steps, "launches_per_round": v[1] / args.steps,
                     "us_per_launch": v[0] * 1e3 / max(1, v[1])} for k, v in kinds.items() if v[1]}

    exp_round = cfg.expansions_per_round()
    value = whole_job_rate(exp_round, world, ms / 1e3)
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
                             ("L2 flushed before every timed round (untimed 512 MB write, then a 512 MB read "
                              "that takes the write-back); the head weights a depth reads (%.0f MB) would fit in L2" %
                              ((wi_bytes_per_depth(cfg) + cfg.d * cfg.d * cfg.bpe) / 1e6))},
            "us_per_round": ms * 1e3,
            # the round's LM-head bytes over the whole round's time (head updates,
            # selection and pruning included), and the LM-head kernel alone
            "lmhead_gbs": lm_bytes_round / (ms / 1e3) / 1e9 if lm_bytes_round else None,
            "lmhead_frac_of_8tbs": lm_bytes_round / (ms / 1e3) / 1e9 / NOMINAL_HBM_GBS if lm_bytes_round else None,
            "lmhead_kernel_frac_of_8tbs": achieved / NOMINAL_HBM_GBS if lm_bytes_round else None,
            "roofline": {"kernel": rl_name, "note": rl_note,
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
