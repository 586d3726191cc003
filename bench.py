#!/usr/bin/env python3
"""Benchmark of the fused CM-ASD logits pass (confidence + verification).

Workload: recipe c3 -- B=64 sequences, K=8 drafted positions, V=128256,
bfloat16 drafter and target logits (Zipf(1.1) profile x4 over a per-row
permutation + 0.5 N(0,1); target = drafter + N(0,1); drafted tokens sampled
from the drafter), SAMPLED rule (Philox acceptance + residual draw).

A step is one call of cmsd_confidence_verify over one batch: the streaming
kernel (every drafter and target logit read once) plus the residual-resample
kernel over the rejected row pair of each sequence.  Two distinct input sets
(2 x 263 MB, each larger than the 129 MB L2) alternate between steps.

Prints one JSON line (rank 0).  --impl reference times the CPU oracle on a
bounded sample of the same workload instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

WORKLOAD = "c3"
METRIC = "confidence+verify logit rows/s at V=128256 (B=64, K=8, bf16 logits)"
UNIT = "rows/s"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


KERNEL_SOURCES = ("cmsd_stream_impl.cuh", "cmsd_device.cuh", "cmsd_internal.h")


def kernel_sources_sha():
    import hashlib
    h = hashlib.sha256()
    for n in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2508_15371_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic():
    """Per-launch DRAM bytes of the streaming kernel from the committed ncu
    summary; None when the kernel sources changed since it was captured."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            d = json.load(f)
        if d.get("sources_sha256_16") != kernel_sources_sha():
            return None
        return d
    except Exception:
        return None


class ClockSampler:
    """nvidia-smi samples (every 100 ms) with host timestamps."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.samples = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", gpu_id, "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception as e:   # noqa: BLE001
            log("clock sampling unavailable:", e)
            return
        self.t = threading.Thread(target=self._read, daemon=True)
        self.t.start()

    def _read(self):
        for line in self.proc.stdout:
            self.samples.append((time.time(), [x.strip() for x in line.split(",")]))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:   # noqa: BLE001
                self.proc.kill()

    def summary(self, t0, t1):
        win = [s for t, s in self.samples if t0 <= t <= t1]
        note = "timed region"
        if len(win) < 3:
            win = [s for t, s in self.samples if t0 - 1.0 <= t <= t1 + 0.2]
            note = "load window around the timed region"
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "window": note}
        sm = [float(s[1]) for s in win if s[1].replace(".", "").isdigit()]
        mx = [float(s[2]) for s in win if s[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for s in win for n, v in zip(names, s[5:9]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(win), "window": note}


def shard_seeds(rank, nsets=2):
    """Seeds of the input sets of one rank: every rank gets its own sequences."""
    from paper_2508_15371_gb300 import workloads as W
    base = W.FULL_SIZES[WORKLOAD]["seed"]
    return [base + 1000 * rank + 100 * j for j in range(nsets)]


def make_sets(rank, nsets=2):
    from paper_2508_15371_gb300 import workloads as W
    return [W.make(WORKLOAD, seed=s) for s in shard_seeds(rank, nsets)]


def max_over_ranks(ms, dist, device):
    """The slowest rank's time (ms); every rank gets the same value."""
    if dist is None:
        return float(ms)
    import torch
    tt = torch.tensor([float(ms)], device=device, dtype=torch.float64)
    dist.all_reduce(tt, op=dist.ReduceOp.MAX)
    return float(tt.item())


def job_rows_per_s(world, rows_per_rank, steps, ms_total):
    """Whole-job throughput: the rows all ranks processed over the slowest rank's time."""
    return world * rows_per_rank * steps / (ms_total * 1e-3)


def oracle_rows_per_s(w, p_dict, budget_s, seeds_from=0, max_rows=None):
    """Time the CPU oracle on whole sequences of w until budget_s is used."""
    import oracle as O
    d64 = O.logits_to_f64(w.draft[seeds_from:seeds_from + 1], w.dtype)
    t64 = O.logits_to_f64(w.target[seeds_from:seeds_from + 1], w.dtype)
    P = O.Params(**p_dict)
    rows = 0
    t0 = time.perf_counter()
    b = 0
    while True:
        O.confidence_verify(d64, t64, w.tokens[seeds_from:seeds_from + 1], P, seed=w.seed, iteration=b)
        rows += w.K
        b += 1
        if time.perf_counter() - t0 >= budget_s or (max_rows and rows >= max_rows):
            break
    dt = time.perf_counter() - t0
    return rows / dt, rows, dt


def run_reference(args):
    """CPU oracle as the reference arm (rank 0 only)."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    import oracle as O
    from paper_2508_15371_gb300 import workloads as W
    w = W.make(WORKLOAD, B=1)
    P = O.Params(k_min=1, k_max=w.K, rule="sampled", beta_rank=0,
                 lam=tuple(float(np.float32(1 / 3)) for _ in range(3)),
                 tau_base=float(np.float32(0.1)))
    d64 = O.logits_to_f64(w.draft, w.dtype)
    t64 = O.logits_to_f64(w.target, w.dtype)
    # calibrate one sequence, then size the per-step sample so the run ends in ~2 minutes
    t0 = time.perf_counter()
    O.confidence_verify(d64, t64, w.tokens, P, seed=w.seed, iteration=0)
    t_seq = time.perf_counter() - t0
    total = args.steps + args.warmup
    rows_per_step = w.K
    if total * t_seq > 120.0:
        rows_per_step = max(1, int(120.0 / total / (t_seq / w.K)))
    k_row = None if rows_per_step >= w.K else np.array([rows_per_step], np.int64)
    for it in range(args.warmup):
        O.confidence_verify(d64, t64, w.tokens, P, seed=w.seed, iteration=it, k_row=k_row)
    t0 = time.perf_counter()
    for it in range(args.steps):
        O.confidence_verify(d64, t64, w.tokens, P, seed=w.seed, iteration=it, k_row=k_row)
    dt = time.perf_counter() - t0
    rows = args.steps * min(rows_per_step, w.K)
    value = rows / dt
    sample = (f"{min(rows_per_step, w.K)} drafted positions (one sequence) of the B=64 K=8 V=128256 "
              f"bf16 workload per step, float64 numpy oracle")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": "c3: B=64 K=8 V=128256 bf16 Zipf(1.1)x4 + 0.5N, target +N, drafted ~ softmax",
                       "rule": "sampled", "sample_rows_per_step": min(rows_per_step, w.K)},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_ours(args):
    import torch

    from paper_2508_15371_gb300 import cmsd

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    # ---- inputs (host generation, then resident in HBM) ---------------------
    t_gen = time.perf_counter()
    sets = make_sets(rank)
    log(f"[rank {rank}] generated {len(sets)} input sets in {time.perf_counter() - t_gen:.1f}s")
    w0 = sets[0]
    B, K, V = w0.B, w0.K, w0.V
    rows = B * K
    alg_bytes = w0.logit_bytes
    p = cmsd.params(K, args.rule)
    dsets = []
    for w in sets:
        dsets.append((cmsd.to_device_logits(w.draft, w.dtype, dev), cmsd.to_device_logits(w.target, w.dtype, dev),
                      torch.from_numpy(w.tokens).to(dev)))
    ws = cmsd.workspace(B, K, V)
    out = {"k_next": torch.empty(B, dtype=torch.int32, device=dev),
           "n_accept": torch.empty(B, dtype=torch.int32, device=dev),
           "out_tokens": torch.empty((B, K), dtype=torch.int32, device=dev)}
    calls = [cmsd.FusedCall(d, t, tk, p, seed=w0.seed, out=out, ws=ws) for d, t, tk in dsets]
    sampled = args.rule == "sampled"
    launches_per_step = 2 if sampled else 1

    # ---- warm-up, clock sampler --------------------------------------------
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:   # noqa: BLE001
        uuid = str(dev.index)
    clocks = ClockSampler(uuid)
    for it in range(args.warmup):
        calls[it % len(calls)](iteration=it)
    torch.cuda.synchronize()
    # keep the GPU loaded before timing so the clock record covers a load window
    t_load = time.time()
    it = 0
    while time.time() - t_load < args.load_window:
        calls[it % len(calls)](iteration=it)
        it += 1
        if it % 200 == 0:
            torch.cuda.synchronize()
    torch.cuda.synchronize()

    # ---- timed region: device-resident inputs -----------------------------
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    t_wall0 = time.time()
    ev0.record()
    for it in range(args.steps):
        calls[it % len(calls)](iteration=it)
    ev1.record()
    torch.cuda.synchronize()
    t_wall1 = time.time()
    if dist:
        dist.barrier()
    ms_total = ev0.elapsed_time(ev1)
    clocks.stop()
    clk = clocks.summary(t_wall0, t_wall1)
    # the same steps again with the library's per-kernel CUDA events (an event
    # between the two kernels serialises them, so this pass is not the one
    # `value` comes from): durations of the streaming and resample kernels
    cmsd.profile_start(args.steps)
    for it in range(args.steps):
        calls[it % len(calls)](iteration=it)
    torch.cuda.synchronize()
    k_ms, r_ms = cmsd.profile_stop(args.steps)
    ms_total = max_over_ranks(ms_total, dist, dev)
    ms_step = ms_total / args.steps
    value = job_rows_per_s(world, rows, args.steps, ms_total)

    # ---- end to end: pinned host inputs, copies inside the timed region ----
    e2e_steps = max(3, min(args.steps, 20))
    host = []
    for w in sets:
        hd = cmsd.to_device_logits(w.draft, w.dtype, "cpu").pin_memory()
        ht = cmsd.to_device_logits(w.target, w.dtype, "cpu").pin_memory()
        hk = torch.from_numpy(w.tokens).pin_memory()
        host.append((hd, ht, hk))
    dbuf = [(torch.empty_like(h[0], device=dev), torch.empty_like(h[1], device=dev),
             torch.empty_like(h[2], device=dev)) for h in host[:1]]
    ecall = cmsd.FusedCall(dbuf[0][0], dbuf[0][1], dbuf[0][2], p, seed=w0.seed, out=out, ws=ws)
    res_host = [torch.empty(B, dtype=torch.int32).pin_memory(), torch.empty((B, K), dtype=torch.int32).pin_memory(),
                torch.empty(B, dtype=torch.int32).pin_memory()]
    h2d = sum(x.numel() * x.element_size() for x in host[0])
    d2h = sum(x.numel() * x.element_size() for x in res_host)

    def e2e_step(j):
        hd, ht, hk = host[j % len(host)]
        dbuf[0][0].copy_(hd, non_blocking=True)
        dbuf[0][1].copy_(ht, non_blocking=True)
        dbuf[0][2].copy_(hk, non_blocking=True)
        o = ecall(iteration=j)
        res_host[0].copy_(o["n_accept"], non_blocking=True)
        res_host[1].copy_(o["out_tokens"], non_blocking=True)
        res_host[2].copy_(o["k_next"], non_blocking=True)

    for j in range(3):
        e2e_step(j)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    for j in range(e2e_steps):
        e2e_step(j)
    e1.record()
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e_ms = max_over_ranks(e2e_ms, dist, dev)
    e2e_value = job_rows_per_s(world, rows, e2e_steps, e2e_ms)

    # ---- roofline of the streaming kernel ----------------------------------
    peak, peak_src = peaks()
    k_mean = statistics.mean(k_ms) if k_ms else float("nan")
    r_mean = statistics.mean(r_ms) if r_ms else 0.0
    achieved = alg_bytes / (k_mean * 1e-3) / 1e9
    tr = ncu_traffic()
    traffic = tr.get("bytes_per_launch") if tr and tr.get("workload") == WORKLOAD and tr.get("rule") == args.rule else None

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return 0

    # ---- decode-loop simulation (rank 0, N = 1 only) -------------------------
    dsim = None
    if world == 1 and not args.no_decode_sim:
        dsim = decode_sim_report()

    # ---- CPU oracle baseline (rank 0, N = 1 only) ---------------------------
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        v, nrows, dt = oracle_rows_per_s(w0, p.as_dict(), budget_s=args.cpu_budget)
        cpu = {"value": v, "unit": UNIT, "cores": 1, "kind": "oracle",
               "sample": f"{nrows} drafted positions ({nrows // K} sequence passes) of this workload, "
                         f"float64 numpy, single thread, {dt:.1f} s"}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "c3: B=64 K=8 V=128256 bf16 logits, Zipf(1.1)x4 profile over a per-row "
                               "permutation + 0.5N(0,1); target = drafter + N(0,1); drafted ~ softmax",
                   "rule": args.rule, "logits": "bf16", "accumulate": "f32",
                   "l2": "inputs larger than L2: 2 alternating input sets of 263 MB each (L2 129 MB)",
                   "parallelism": f"dp{world} (independent batches per GPU)" if world > 1 else "single GPU"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "kernel": "stream_kernel (fused confidence + verify pass)",
                     "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured" else "fallback 6800 GB/s",
                     "algorithmic_bytes_per_launch": alg_bytes, "kernel_ms": k_mean,
                     "kernel_timing": "CUDA events around each streaming-kernel launch, averaged over a "
                                      "second pass of the same steps"},
        "hbm_gbs_step": alg_bytes / (ms_step * 1e-3) / 1e9,
        "resample_ms": r_mean,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "steps": e2e_steps},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
    }
    if dsim is not None:
        line["decode_sim"] = dsim
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def decode_sim_report(B=32, K=16, V=32000, iterations=512):
    """Algorithm 1 as a decode loop over device-generated f32 logits: k_next of
    each iteration is the next iteration's k_row.  Timed with CUDA events over
    all iterations (logit generation included)."""
    import torch
    from paper_2508_15371_gb300 import cmsd, decode_sim
    p = cmsd.params(K, "sampled")
    sim = decode_sim.DecodeSim(B, K, V, iterations, p, seed=4)
    for it in range(3):
        sim.step(it)
    torch.cuda.synchronize()
    sim = decode_sim.DecodeSim(B, K, V, iterations, p, seed=4)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for it in range(iterations):
        sim.step(it)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1)
    hist = {"k": sim.hist_k.cpu().numpy(), "n_accept": sim.hist_n.cpu().numpy()}
    s = decode_sim.summarize(hist)
    s.update({"workload": f"B={B} K_max={K} V={V} f32, {iterations} iterations, sampled rule, AR(1) spike heights",
              "ms_per_iteration": ms / iterations, "rows_per_s": s["rows"] / (ms * 1e-3),
              "timing": "CUDA events over the loop, device logit generation included"})
    return s


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--rule", choices=["sampled", "paper"], default="sampled")
    ap.add_argument("--cpu-budget", type=float, default=10.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode-sim", action="store_true", help="skip the decode-loop simulation report")
    ap.add_argument("--load-window", type=float, default=0.8,
                    help="seconds of untimed steps just before the timed region (clock sampling)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
