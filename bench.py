#!/usr/bin/env python3
"""Benchmark of FadeMem's per-segment memory step on GB300 (one JSON line).

Workload (Wan2.1-1.3B shaped, one layer, bf16): 12 heads, head_dim 128, 1560
tokens per latent frame, 3-frame segments (4680 query tokens), budget 21
entries, beta 0.3, first-frame anchor on, synthetic AR(1) K/V (rho 0.9) and
N(0,1) queries.  The memory is first brought to steady state (21 entries, 3
merges per segment).  One step = insert the segment's 3 frames + device
schedule + fused consolidation + attention of the 4680 queries over the 21
consolidated entries (32,760 keys per head).  In steady state the schedule of
each pass is computed ahead, inside the previous consolidation kernel.

Metric: query tokens per second per layer over (attend + consolidate) time.
`value` times the device-resident step with CUDA events, L2 flushed (256 MiB
write, then 256 MiB read) before every step and excluded from the step time.  `e2e` times the
same step through the C ABI with pinned host buffers: host->device copy of
K, V and Q, the three calls, device->host copy of the output.

--impl reference times the fp64 CPU oracle on this machine's cores on a
bounded sample of the same workload (see cpu_baseline).
"""
from __future__ import annotations

import argparse
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

H, D, N, F, M, BETA = 12, 128, 1560, 3, 21, 0.3
LQ = F * N
WORKLOAD = "wan2.1-1.3b-shaped single layer: H=12 D=128 N=1560 frames/segment=3 Lq=4680 M=21 beta=0.3 bf16"
# --workload: the headline (default) and the per-layer unit of the 14B model (H=40), timed as one
# attend + one consolidate at that shape.
WORKLOADS = {
    "wan1.3b": (12, WORKLOAD),
    "wan14b": (40, "wan2.1-14b-shaped single layer (one layer of the 40-layer model): H=40 D=128 N=1560 "
                   "frames/segment=3 Lq=4680 M=21 beta=0.3 bf16"),
}
METRIC = "query tokens/s per layer (attend+consolidate)"


# Nominal GB300 HBM3e bandwidth (context only; fractions are taken against measured peaks).
NOMINAL_HBM_GBS = 7900.0


def _peaks():
    """(HBM GB/s, bf16 burst TFLOP/s, bf16 sustained TFLOP/s, kind): the measured copy and
    cuBLAS figures of this machine, else the fallback figures of an earlier GB300."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as fh:
            p = json.load(fh)
        return (float(p["hbm_gbs"]), float(p["bf16_tflops"]),
                float(p.get("bf16_tflops_sustained", p["bf16_tflops"])), "measured")
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


def _profiled_traffic(profile: str, source: str):
    """DRAM bytes per launch from a committed ncu summary, or None if the kernel
    source changed since those counters were taken (hash recorded in the summary)."""
    if H != 12:
        return None  # the committed captures are of the default workload
    import hashlib
    try:
        text = open(os.path.join(ROOT, "profiles", profile)).read()
        want = re.search(r"source_sha256_prefix:\s*([0-9a-f]+)", text).group(1)
        traffic = int(re.search(r"traffic_bytes_per_launch:\s*(\d+)", text).group(1))
        have = hashlib.sha256(open(os.path.join(ROOT, source), "rb").read()).hexdigest()[:len(want)]
        return traffic if have == want else None
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        rows = []
        try:
            for ln in open(self.path):
                parts = [x.strip() for x in ln.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        except Exception:
            pass
        finally:
            try:
                os.unlink(self.path)
            except Exception:
                pass
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower().startswith("active")})
        busy = sorted(sm)[len(sm) // 4:] if sm else []  # samples under load (drop idle ramp)
        return {"sm_mhz": statistics.median(busy) if busy else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(rows)}


def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def max_over_ranks(x: float, device) -> float:
    """The largest value over all ranks (the slowest replica sets the job's time).

    Replicas only: the memory step has no data-path exchange (heads and layers are
    independent and the schedule depends on frame counts alone), so each rank runs
    its own memory and the only collective is this timing reduction.
    """
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: float, step_ms: float, world: int) -> float:
    """Units processed by all ranks per second, timed by the slowest rank (weak scaling)."""
    return world * units_per_rank / (step_ms / 1e3)


def _segment_inputs(seed, n_sets, device):
    """n_sets distinct (K, V, Q) segment inputs, AR(1) K/V across the sets' frames."""
    from synth import KIND_K, KIND_V, DeviceAR1, device_queries
    gk = DeviceAR1((N, H, D), seed, KIND_K, 0, device=device)
    gv = DeviceAR1((N, H, D), seed, KIND_V, 0, device=device)
    sets = []
    for s in range(n_sets):
        K = torch.stack([gk.next() for _ in range(F)]).contiguous()
        V = torch.stack([gv.next() for _ in range(F)]).contiguous()
        Q = device_queries((LQ, H, D), seed, 0, s, device=device)
        sets.append((K, V, Q))
    return sets


def run_cuda(args):
    from paper_2606_10671_gb300 import FadeMem
    from paper_2606_10671_gb300 import build as _b
    ws, rank, local = _dist()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    _b.build_library()

    mem = FadeMem(M, H, D, N, num_layers=1, beta=BETA, anchor=True, dtype=torch.bfloat16, device=dev)
    n_sets = 4
    sets = _segment_inputs(1000 + rank, n_sets, dev)
    out = torch.empty((LQ, H, D), dtype=torch.bfloat16, device=dev)
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size
    flush_bytes = max(2 * l2, 256 << 20)
    flush = torch.empty(flush_bytes, dtype=torch.uint8, device=dev)
    flush_read = torch.ones(flush_bytes // 4, dtype=torch.float32, device=dev)

    def flush_l2():
        # Write a buffer larger than L2, then read another one: L2 ends up holding
        # only clean lines of unrelated data, so the step neither hits in L2 nor
        # pays the write-back of the flush's own dirty lines.
        flush.zero_()
        flush_read.sum()
    stream = torch.cuda.current_stream(dev)

    # Steady state: 8 segments of 3 frames fill the 21-entry budget and start merging.
    for s in range(8):
        K, V, _ = sets[s % n_sets]
        mem.insert(0, K, V)
        mem.consolidate()

    def step(i):
        K, V, Q = sets[i % n_sets]
        mem.insert(0, K, V)
        mem.consolidate()
        return Q

    for i in range(args.warmup):
        Q = step(i)
        mem.attend(0, Q, out)
    torch.cuda.synchronize()
    mem.device_status()

    # algorithmic bytes of the consolidation: every plan source read once, every changed slot written once
    block_bytes = 2 * N * H * D * 2  # K + V of one entry of one layer, bf16
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    blocks0, passes0, launches0 = mem.stats()
    if ws > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    region0 = torch.cuda.Event(enable_timing=True)
    region1 = torch.cuda.Event(enable_timing=True)
    with ClockSampler(torch.cuda.current_device() if "CUDA_VISIBLE_DEVICES" not in os.environ else local) as clk:
        region0.record(stream)
        for i in range(args.steps):
            flush_l2()
            e0, e1, e2 = ev[i]
            e0.record(stream)
            Q = step(args.warmup + i)
            e1.record(stream)
            mem.attend(0, Q, out)
            e2.record(stream)
        region1.record(stream)
        torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    clocks = clk.summary()
    t_cons = [ev[i][0].elapsed_time(ev[i][1]) for i in range(args.steps)]
    t_attn = [ev[i][1].elapsed_time(ev[i][2]) for i in range(args.steps)]
    blocks1, passes1, launches1 = mem.stats()
    # Host cost of enqueuing one step (insert + consolidate + attend through the binding and
    # the ABI), measured from an idle GPU on few enough steps that the launch queue never fills.
    torch.cuda.synchronize()
    host_us = []
    for i in range(20):
        h0 = time.perf_counter()
        Q = step(i)
        mem.attend(0, Q, out)
        host_us.append((time.perf_counter() - h0) * 1e6)
    torch.cuda.synchronize()
    mem.device_status()
    step_ms = max_over_ranks((sum(t_cons) + sum(t_attn)) / args.steps, dev)
    value = whole_job_rate(LQ, step_ms, ws)

    hbm_peak, bf16_peak, bf16_sustained, peak_kind = _peaks()
    attn_ms = statistics.mean(t_attn)
    cons_ms = statistics.mean(t_cons)
    Lk = M * N
    flops = 4.0 * LQ * Lk * H * D
    attn_tflops = flops / (attn_ms / 1e3) / 1e12
    # Mean per step (one fademem_consolidate call of 3 frames = one pass).  It falls slowly over a
    # long run: anchor merges, which move no bytes, grow more frequent as the history lengthens.
    cons_bytes = (blocks1 - blocks0) * block_bytes / args.steps
    cons_gbs = cons_bytes / (cons_ms / 1e3) / 1e9

    # End to end through the C ABI with host buffers: fademem_step_host copies each step's
    # K, V and Q in from pinned host memory (on the library's copy stream, overlapping the
    # previous step's work), inserts, consolidates, attends and copies the output back to
    # the host.  Timed as one region over the steps; no L2 flush is needed because every
    # step streams the 201 MB memory, more than L2 holds.
    hK = [s[0].cpu().pin_memory() for s in sets]
    hV = [s[1].cpu().pin_memory() for s in sets]
    hQ = [s[2].cpu().pin_memory() for s in sets]
    hO = [torch.empty((LQ, H, D), dtype=torch.bfloat16).pin_memory() for _ in range(2)]
    for i in range(args.warmup):
        j = i % n_sets
        mem.step_host([hK[j]], [hV[j]], hQ[j], hO[i % 2])
    torch.cuda.synchronize()
    if ws > 1:
        torch.distributed.barrier()
    e2e0 = torch.cuda.Event(enable_timing=True)
    e2e1 = torch.cuda.Event(enable_timing=True)
    e2e0.record(stream)
    for i in range(args.steps):
        j = i % n_sets
        mem.step_host([hK[j]], [hV[j]], hQ[j], hO[i % 2])
    e2e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e2e0.elapsed_time(e2e1) / args.steps, dev)
    h2d = sum(x.numel() * x.element_size() for x in (hK[0], hV[0], hQ[0]))
    d2h = hO[0].numel() * hO[0].element_size()
    mem.device_status()

    line = {
        "metric": METRIC,
        "value": round(value, 1),
        "unit": "tokens/s",
        "n_gpus": ws,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": round(step_ms, 4),
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic (AR(1) K/V rho=0.9, N(0,1) Q; no model weights)",
        "config": {"workload": WORKLOAD, "steady_state_entries": M, "keys_per_head": Lk,
                   "l2": "flushed before every step (256 MiB write, then 256 MiB read of another buffer), "
                         "flush excluded from step time",
                   "parallelism": f"replicas x{ws} (one independent memory per GPU)"},
        "gpu_launches": launches1 - launches0,  # counted by the library
        "host_enqueue_us_per_step": round(statistics.median(host_us), 1),  # binding + ABI calls, GPU idle
        "roofline": {"bound": "tensor", "kernel": "attend_tc_kernel", "achieved": round(attn_tflops, 1),
                     "peak": bf16_peak, "unit": "TFLOP/s", "frac": round(attn_tflops / bf16_peak, 4),
                     "peak_kind": f"{peak_kind} bf16 burst",
                     "peak_sustained": bf16_sustained, "frac_of_sustained": round(attn_tflops / bf16_sustained, 4),
                     "traffic": _profiled_traffic("attend_tc_wan13b.md", "paper_2606_10671_gb300/csrc/attend_tc.cu"),
                     "flops_per_launch": flops, "ms_per_launch": round(attn_ms, 4)},
        "consolidate": {"bound": "hbm", "achieved": round(cons_gbs, 1), "peak": hbm_peak, "unit": "GB/s",
                        "frac": round(cons_gbs / hbm_peak, 4), "bytes_per_step": round(cons_bytes),
                        "frac_of_nominal": round(cons_gbs / NOMINAL_HBM_GBS, 4), "nominal_gbs": NOMINAL_HBM_GBS,
                        "ms_per_step": round(cons_ms, 4),
                        "blocks_per_step": round((blocks1 - blocks0) / args.steps, 3),
                        "passes_per_step": round((passes1 - passes0) / args.steps, 3),
                        "note": "event time of the fademem_consolidate call (in steady state the consolidation "
                                "kernel alone: the next pass is scheduled inside it); algorithmic bytes from the "
                                "device's own count of blocks moved over the timed steps",
                        "traffic": _profiled_traffic("consolidate_wan13b.md",
                                                     "paper_2606_10671_gb300/csrc/consolidate.cu")},
        "region_ms": round(region0.elapsed_time(region1), 3),
        "clocks": clocks,
        "e2e": {"value": round(whole_job_rate(LQ, e2e_ms, ws), 1), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": round(e2e_ms, 4),
                "api": "fademem_step_host (pinned host K, V, Q in; out back to pinned host memory), "
                       "timed as one region over the steps"},
    }
    if args.rope_pairs > 0:
        line["rope"] = _measure_rope(args, sets, out, flush_l2, stream, dev, cons_ms, hbm_peak)
    if rank == 0 and ws == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(args.cpu_queries)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if ws > 1:
        torch.distributed.destroy_process_group()


def _measure_rope(args, sets, out, flush_l2, stream, dev, cons_ms_plain, hbm_peak):
    """The same workload with temporal RoPE handling on (Sec. 3.3, "Boundary and positional
    handling"; Wan2.1's temporal band of 22 complex pairs): per step the consolidation call
    now also runs the re-phase kernel, which writes the re-indexed attention keys of every
    entry (read stored K + write K_att: count * N * H * D * 2 bytes each way)."""
    from paper_2606_10671_gb300 import FadeMem
    mem = FadeMem(M, H, D, N, num_layers=1, beta=BETA, anchor=True, dtype=torch.bfloat16, device=dev,
                  rope_pairs=args.rope_pairs)
    for s_ in range(8):
        K, V, _ = sets[s_ % len(sets)]
        mem.insert(0, K, V)
        mem.consolidate()
    steps = max(20, args.steps // 6)
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    for i in range(steps + 3):
        K, V, Q = sets[i % len(sets)]
        flush_l2()
        if i >= 3:
            ev[i - 3][0].record(stream)
        mem.insert(0, K, V)
        mem.consolidate()
        if i >= 3:
            ev[i - 3][1].record(stream)
        mem.attend(0, Q, out)
        if i >= 3:
            ev[i - 3][2].record(stream)
    torch.cuda.synchronize()
    mem.device_status()
    cons = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    attn = statistics.mean(e[1].elapsed_time(e[2]) for e in ev)
    rephase_bytes = 2 * M * N * H * D * 2
    re_ms = max(cons - cons_ms_plain, 1e-6)
    return {"rope_pairs": args.rope_pairs, "steps": steps, "consolidate_ms_per_step": round(cons, 4),
            "attend_ms_per_step": round(attn, 4), "value": round(LQ / ((cons + attn) / 1e3), 1), "unit": "tokens/s",
            "rephase_bytes_per_step": rephase_bytes,
            "rephase_ms_est": round(re_ms, 4),
            "rephase_frac_est": round(rephase_bytes / (re_ms / 1e3) / 1e9 / hbm_peak, 4),
            "note": "rephase time estimated as this consolidate time minus the RoPE-off one; its own ncu "
                    "duration is in profiles/"}


class OracleStep:
    """The fp64 oracle, as it stands, stepping the same workload on this host's cores.

    The memory is warmed once (M + 3 frames: full budget, merging).  One step
    inserts a segment's 3 frames (a full steady-state consolidation of all 12
    heads and every token, timed) and attends a bounded sample of the 4680
    query rows over all 12 heads and 32,760 keys per head (timed); the
    attention time is scaled to the 4680 rows.  Frame generation is not timed.
    """

    def __init__(self, seed: int = 7):
        from oracle import OracleMemory
        from synth import KIND_K, KIND_V, HostAR1
        self.mem = OracleMemory(M, BETA, anchor=True, elems=N * H * D)
        self.gk = HostAR1((N, H, D), seed, KIND_K)
        self.gv = HostAR1((N, H, D), seed, KIND_V)
        self.seed = seed
        self.steps = 0
        for _ in range(M + 3):
            self.mem.insert(self._frame(self.gk), self._frame(self.gv))

    @staticmethod
    def _frame(g):
        return torch.from_numpy(g.next()).to(torch.bfloat16).double().numpy()

    def step(self, n_queries: int):
        from synth import host_queries
        new = [(self._frame(self.gk), self._frame(self.gv)) for _ in range(F)]
        Q = torch.from_numpy(host_queries((n_queries, H, D), self.seed, 0, self.steps)).to(
            torch.bfloat16).double().numpy()
        self.steps += 1
        t0 = time.perf_counter()
        for K, V in new:
            self.mem.insert(K, V)
        t_cons = time.perf_counter() - t0
        t0 = time.perf_counter()
        self.mem.attend(Q, N, H, D)
        t_attn = time.perf_counter() - t0
        return t_cons, t_attn, t_cons + t_attn * (LQ / n_queries)


def _oracle_sample(n_queries: int) -> str:
    return (f"fp64 C oracle: one full 3-frame consolidation (12 heads x 1560 tokens) + attention of "
            f"{n_queries}/{LQ} query rows x {H} heads over {M * N} keys, scaled to {LQ} rows")


def cpu_baseline(n_queries: int = 2340):
    """One oracle step on a bounded sample (about 10 s of CPU work at the default)."""
    from oracle import oracle_num_threads
    o = OracleStep()
    t_cons, t_attn, step_s = o.step(n_queries)
    return {"value": round(LQ / step_s, 3), "unit": "tokens/s", "cores": oracle_num_threads(), "kind": "oracle",
            "sample": _oracle_sample(n_queries), "seconds_measured": round(t_cons + t_attn, 2)}


def run_reference(args):
    """The oracle as the reference arm: each step a bounded sample of the same workload."""
    from oracle import oracle_num_threads
    ws, rank, _ = _dist()
    if rank != 0:
        return
    nq = args.ref_queries
    o = OracleStep()
    for _ in range(args.warmup):
        o.step(nq)
    times = [o.step(nq)[2] for _ in range(args.steps)]
    step_s = statistics.mean(times)
    value = LQ / step_s
    line = {"impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": "tokens/s", "n_gpus": ws,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(step_s * 1e3, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (AR(1) K/V rho=0.9, N(0,1) Q)",
            "config": {"workload": WORKLOAD},
            "cpu_baseline": {"value": round(value, 3), "unit": "tokens/s", "cores": oracle_num_threads(),
                             "kind": "oracle", "sample": _oracle_sample(nq)},
            "e2e": {"value": round(value, 3), "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["cuda", "reference"], default="cuda")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="wan1.3b")
    ap.add_argument("--rope-pairs", type=int, default=22,
                    help="also time the workload with temporal RoPE handling on this many pairs (0: skip)")
    ap.add_argument("--cpu-queries", type=int, default=2340, help="query rows of the cpu_baseline sample")
    ap.add_argument("--ref-queries", type=int, default=240, help="query rows per --impl reference step")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    global H, WORKLOAD
    H, WORKLOAD = WORKLOADS[args.workload]
    if args.impl == "reference":
        run_reference(args)
    else:
        run_cuda(args)


if __name__ == "__main__":
    main()
