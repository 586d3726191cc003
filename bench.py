#!/usr/bin/env python3
"""Benchmark of the fused CM-ASD logits pass (confidence + verification).

Headline workload: recipe c3 -- B=64 sequences, K=8 drafted positions,
V=128256, bfloat16 drafter and target logits (Zipf(1.1) profile x4 over a
per-row permutation + 0.5 N(0,1); target = drafter + N(0,1); drafted tokens
sampled from the drafter), SAMPLED rule (Philox acceptance + residual draw).

A step is one call of cmsd_confidence_verify over one batch: the streaming
kernel (every drafter and target logit read once) plus the residual draw at
each sequence's rejected position (a cluster of CTAs per row: the target row
again, and the drafter logits of the few groups the bound keeps).  Two
distinct input sets
(2 x 263 MB, each larger than the 129 MB L2) alternate between steps.

Besides the headline, one JSON line carries (rank 0, one GPU): the other
workloads (c1 latency, c2, c4, c3 under the paper's own rule), the decode-loop
simulation (c5) with its generation and pass timed apart and the ablation
variants of Table III, the CPU oracle timed on all host cores with a live
parity check of its sample, and the flagged-decision counts of the full-size
parity record.  --impl reference times the CPU oracle instead.
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
C3_DESC = ("c3: B=64 K=8 V=128256 bf16 logits, Zipf(1.1)x4 profile over a per-row permutation + 0.5N(0,1); "
           "target = drafter + N(0,1); drafted ~ softmax")


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


def measured_peaks():
    """MEASURED_PEAKS.json as a dict ({} when it is absent)."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except Exception:
        return {}


LMHEAD_SOURCES = ("cmsd_lmhead.cu", "cmsd_stream_impl.cuh", "cmsd_device.cuh", "cmsd_internal.h")


def kernel_sources_sha(sources=None):
    import hashlib
    h = hashlib.sha256()
    for n in (KERNEL_SOURCES if sources is None else sources):
        with open(os.path.join(ROOT, "paper_2508_15371_gb300", "csrc", n), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def ncu_traffic(workload, rule):
    """Per-launch DRAM bytes of the streaming kernel from the committed ncu
    summary for this workload and rule; None when the kernel sources changed
    since it was captured."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            recs = json.load(f)
        recs = recs if isinstance(recs, list) else [recs]
        for d in recs:
            if d.get("workload") == workload and d.get("rule") == rule and \
                    d.get("kernel", "").startswith("stream_kernel") and \
                    d.get("sources_sha256_16") == kernel_sources_sha():
                return d.get("bytes_per_launch")
    except Exception:
        pass
    return None


def parity_record(workload, rule):
    """Flagged decisions and largest deviations of the full-size parity test
    (profiles/parity_full_size.json, written from the GPU tests' records)."""
    try:
        with open(os.path.join(ROOT, "profiles", "parity_full_size.json")) as f:
            d = json.load(f)
        for r in d.get("records", []):
            if r.get("workload") == workload and r.get("rule") == rule:
                out = {k: r[k] for k in ("sequences", "decisions", "flagged", "max_abs_err") if k in r}
                out["current_kernels"] = d.get("sources_sha256_16") == kernel_sources_sha()
                return out
    except Exception:
        pass
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


def stats_ms(xs):
    xs = sorted(xs)
    return {"median": statistics.median(xs), "p10": float(np.percentile(xs, 10)),
            "p90": float(np.percentile(xs, 90)), "min": xs[0], "max": xs[-1], "n": len(xs)}


def time_total(torch, calls, nsteps, it0=0):
    """Two CUDA events around nsteps steps on the launching stream: total ms."""
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for i in range(nsteps):
        calls[i % len(calls)](iteration=it0 + i)
    e1.record()
    torch.cuda.synchronize()
    return e0.elapsed_time(e1)


def time_steps(torch, calls, nsteps, it0=0):
    """CUDA events around every step on the launching stream: (total ms, per-step ms).
    An event between steps costs about 2 us of device time per step on this
    path, so the spread comes from this pass and throughput from time_total."""
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(nsteps + 1)]
    ev[0].record()
    for i in range(nsteps):
        calls[i % len(calls)](iteration=it0 + i)
        ev[i + 1].record()
    torch.cuda.synchronize()
    return ev[0].elapsed_time(ev[-1]), [ev[i].elapsed_time(ev[i + 1]) for i in range(nsteps)]


def kernel_times(cmsd, torch, calls, nsteps):
    """The library's per-kernel events (streaming, resample) over nsteps calls."""
    cmsd.profile_start(nsteps)
    for i in range(nsteps):
        calls[i % len(calls)](iteration=i)
    torch.cuda.synchronize()
    return cmsd.profile_stop(nsteps)


# ---------------------------------------------------------------- CPU oracle

def _oracle_seq_task(task):
    """Oracle over whole sequences (worker process): returns rows, seconds and
    the per-sequence results used by the live parity check."""
    draft, target, tokens, dtype, pdict, seed, iteration, b_index = task
    import oracle as O
    P = O.Params(**pdict)
    t0 = time.perf_counter()
    res = []
    for j, b in enumerate(b_index):
        d = O.logits_to_f64(draft[j:j + 1], dtype)
        t = O.logits_to_f64(target[j:j + 1], dtype)
        r = O.confidence(d, P)
        v = O.verify_sequence(d[0], t[0], tokens[j], r.conf[0], d.shape[1], P, seed, int(b), iteration)
        res.append({"b": int(b), "k_next": int(r.k_next[0]), "k_flag": bool(r.k_flag[0]),
                    "n_accept": int(v["n_accept"]), "n_flag": bool(v["n_flag"]),
                    "out_tokens": v["out_tokens"].tolist(), "tok_flag": bool(v["tok_flag"]),
                    "conf": r.conf[0].tolist()})
    return len(b_index) * draft.shape[1], time.perf_counter() - t0, res


def _seq_task(w, b, pdict, seed, iteration):
    return (np.ascontiguousarray(w.draft[b:b + 1]), np.ascontiguousarray(w.target[b:b + 1]),
            np.ascontiguousarray(w.tokens[b:b + 1]), w.dtype, pdict, seed, iteration, [b])


def oracle_pool_run(w, pdict, seed, iteration, budget_s, procs):
    """Time the oracle on whole sequences of w over `procs` worker processes
    (spawned, so no worker is a fork of this CUDA process) for about
    budget_s; returns (rows/s, rows, seconds, per-sequence results)."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs) as pool:
        pool.map(_oracle_seq_task, [_seq_task(w, 0, pdict, seed, iteration)] * procs)   # workers warm
        t0 = time.perf_counter()
        out = pool.map(_oracle_seq_task, [_seq_task(w, b % w.B, pdict, seed, iteration) for b in range(procs)])
        t_round = time.perf_counter() - t0
        rounds = max(0, int((budget_s - t_round) / max(t_round, 1e-3)))
        more = [_seq_task(w, (procs + j) % w.B, pdict, seed, iteration) for j in range(rounds * procs)]
        out += pool.map(_oracle_seq_task, more)
        dt = time.perf_counter() - t0
    rows = sum(x[0] for x in out)
    seen, results = set(), []
    for x in out:
        for r in x[2]:
            if r["b"] not in seen:
                seen.add(r["b"])
                results.append(r)
    return rows / dt, rows, dt, results


def live_parity(results, g, K):
    """Compare the oracle's per-sequence results with the GPU's outputs:
    flagged decisions and mismatches (outside the flagged ones)."""
    flagged = mism = 0
    maxc = 0.0
    for r in results:
        b = r["b"]
        maxc = max(maxc, float(np.max(np.abs(g["conf"][b].astype(np.float64) - np.array(r["conf"])))))
        if r["k_flag"]:
            flagged += 1
        elif g["k_next"][b] != r["k_next"]:
            mism += 1
        if r["n_flag"]:
            flagged += 1
        elif g["n_accept"][b] != r["n_accept"]:
            mism += 1
        if r["tok_flag"]:
            flagged += 1
        elif list(g["out_tokens"][b]) != r["out_tokens"]:
            mism += 1
    return {"sequences": len(results), "decisions": 3 * len(results), "flagged": flagged,
            "mismatches": mism, "max_abs_err_conf": maxc}


def host_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:   # pragma: no cover
        return os.cpu_count() or 1


# ---------------------------------------------------------------- reference arm

def run_reference(args):
    """CPU oracle as the reference arm (rank 0 only), on all host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    os.environ.setdefault("OMP_NUM_THREADS", "1")
    from paper_2508_15371_gb300 import workloads as W
    w = W.make(WORKLOAD, B=16)
    pdict = dict(k_min=1, k_max=w.K, rule="sampled", beta_rank=0,
                 lam=tuple(float(np.float32(1 / 3)) for _ in range(3)), tau_base=float(np.float32(0.1)))
    procs = max(1, min(16, host_cores()))
    # each step: one whole sequence per worker, timed as a batch
    total = args.steps + args.warmup
    times = []
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    with ctx.Pool(procs) as pool:
        for st in range(total):
            tasks = [_seq_task(w, (st * procs + j) % w.B, pdict, w.seed, st) for j in range(procs)]
            t0 = time.perf_counter()
            pool.map(_oracle_seq_task, tasks)
            dt = time.perf_counter() - t0
            if st >= args.warmup:
                times.append(dt)
            if sum(times) > 150.0:
                break
    rows = len(times) * procs * w.K
    dt = sum(times)
    value = rows / dt
    sample = (f"{procs} whole sequences (K={w.K} positions each, one per worker) of the B=64 K=8 V=128256 bf16 "
              f"workload per step, float64 numpy oracle, {len(times)} steps")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": len(times), "warmup": args.warmup, "ms_per_step": 1e3 * dt / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": C3_DESC, "rule": "sampled", "sample_rows_per_step": procs * w.K},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": procs, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------- other workloads

def bench_workload(cmsd, torch, dev, name, rule, steps, peak, nsets=1, graph_latency=False, **size):
    """Device-resident timing of one workload: per-step times (median and
    spread), the streaming kernel's time and its HBM roofline."""
    from paper_2508_15371_gb300 import workloads as W
    base = W.FULL_SIZES[name]["seed"]
    sets = [W.make(name, seed=base + 100 * j, **size) for j in range(nsets)]
    w0 = sets[0]
    p = cmsd.params(w0.K, rule)
    ws = cmsd.workspace(w0.B, w0.K, w0.V)
    out = {"k_next": torch.empty(w0.B, dtype=torch.int32, device=dev),
           "n_accept": torch.empty(w0.B, dtype=torch.int32, device=dev),
           "out_tokens": torch.empty((w0.B, w0.K), dtype=torch.int32, device=dev)}
    calls = []
    for w in sets:
        d = cmsd.to_device_logits(w.draft, w.dtype, dev)
        t = cmsd.to_device_logits(w.target, w.dtype, dev)
        tk = torch.from_numpy(w.tokens).to(dev)
        calls.append(cmsd.FusedCall(d, t, tk, p, seed=w.seed, out=out, ws=ws))
    desc = f"{name}: B={w0.B} K={w0.K} V={w0.V} {w0.dtype}"
    K, V, rows, alg = w0.K, w0.V, w0.rows, w0.logit_bytes
    es = 4 if w0.dtype == "f32" else 2
    del sets, w0
    for i in range(5):
        calls[i % len(calls)](iteration=i)
    torch.cuda.synchronize()
    total = time_total(torch, calls, steps)
    _, per = time_steps(torch, calls, steps)
    k_ms, r_ms = kernel_times(cmsd, torch, calls, steps)
    n = out["n_accept"].cpu().numpy()
    rejected = int((n < K).sum()) if rule == "sampled" else 0
    st = stats_ms(per)
    km = statistics.median(k_ms)
    res = {"workload": desc, "rule": rule,
           "rows_per_s": rows * steps / (total * 1e-3), "ms_per_step": total / steps, "step_ms": st,
           "kernel_ms": km, "resample_ms": statistics.median(r_ms) if rule == "sampled" else 0.0,
           "algorithmic_bytes": alg, "kernel_gbs": alg / (km * 1e-3) / 1e9,
           "kernel_frac": alg / (km * 1e-3) / 1e9 / peak,
           "step_gbs": (alg + rejected * V * es) / (total / steps * 1e-3) / 1e9,   # + the rejected target rows
           "l2": "inputs larger than L2" if alg > 129e6 else "L2-resident (inputs smaller than L2)",
           "traffic": ncu_traffic(name, rule), "parity": parity_record(name, rule)}
    res["step_frac"] = res["step_gbs"] / peak
    if graph_latency:
        # launch cost removed: the same call captured 20 times in a CUDA graph
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            for i in range(20):
                calls[0](iteration=i)
        g.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(10):
            g.replay()
        e1.record()
        torch.cuda.synchronize()
        res["latency_us_graph"] = e0.elapsed_time(e1) / 200 * 1e3
        res["latency_us_launch"] = st["median"] * 1e3
    del calls
    torch.cuda.empty_cache()
    return res


def lmhead_traffic():
    """Per-launch DRAM bytes of the LM-head GEMM kernel from the committed ncu
    summary; None when its sources changed since it was captured."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            for d in json.load(f):
                if d.get("workload") == "lmhead" and \
                        d.get("sources_sha256_16") == kernel_sources_sha(LMHEAD_SOURCES):
                    return d.get("bytes_per_launch")
    except Exception:
        pass
    return None


def lmhead_report(cmsd, torch, hbm_peak, R=64, d=2048, V=128256, calls=100):
    """The drafter's LM head fused with the confidence signals
    (cmsd_lmhead_confidence): R hidden rows of a d-wide drafter through a
    [V, d] bf16 head.  Timed with CUDA events over `calls` back-to-back calls
    (the 525 MB weight is larger than L2); beside it, the same result unfused:
    a cuBLAS bf16 GEMM (torch.matmul) writing the logits, then
    cmsd_confidence over them.  Parity: the oracle on 8 of the rows."""
    from paper_2508_15371_gb300 import workloads as W
    w = W.make_lmhead(R=R, d=d, V=V, seed=7)
    h = torch.from_numpy(w.hidden.view(np.int16)).cuda()
    wt = torch.from_numpy(w.weight.view(np.int16)).cuda()
    p = cmsd.params(1)
    ws = cmsd.lmhead_workspace(R, d, V)
    out = {n: torch.empty(R, dtype=torch.float32, device="cuda") for n in ("H", "margin", "conf", "lse")}
    out["argmax"] = torch.empty(R, dtype=torch.int32, device="cuda")
    hb, wb = h.view(torch.bfloat16), wt.view(torch.bfloat16)
    lg = torch.empty((R, V), dtype=torch.bfloat16, device="cuda")
    cws = cmsd.workspace(R, 1, V)
    co = {n: torch.empty((R, 1), dtype=torch.float32, device="cuda") for n in ("H", "margin", "conf", "lse")}
    co["argmax"] = torch.empty((R, 1), dtype=torch.int32, device="cuda")
    co["k_next"] = torch.empty(R, dtype=torch.int32, device="cuda")

    def fused():
        cmsd.lmhead_confidence(h, wt, p=p, out=out, ws=ws)

    def gemm():
        torch.matmul(hb, wb.t(), out=lg)

    def unfused():
        gemm()
        cmsd.confidence(lg.view(R, 1, V), p=p, out=co, ws=cws)

    def timed(fn):
        for _ in range(5):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        for _ in range(calls):
            fn()
        e1.record()
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / calls

    ms_f, ms_g, ms_u = timed(fused), timed(gemm), timed(unfused)
    g = {k: v.cpu().numpy() for k, v in out.items()}
    import oracle as O
    rows = np.arange(0, R, max(1, R // 8))
    P = O.Params(lam=tuple(p.lam), beta_sig=p.beta_sig)
    o = O.lm_head_confidence(w.hidden[rows], w.weight, P)
    habs = np.abs(O.bf16_bits_to_f64(w.hidden[rows]))
    eps = d * 2.0 ** -23 * (habs @ np.abs(O.bf16_bits_to_f64(w.weight)).T).max(axis=1)
    clear = o["margin"] > 2 * eps
    bytes_ = V * d * 2 + R * d * 2
    flops = 2.0 * R * d * V
    achieved = bytes_ / (ms_f * 1e-3) / 1e9
    tflops = flops / (ms_f * 1e-3) / 1e12
    tpeak = measured_peaks().get("bf16_tflops")
    return {
        "workload": f"R={R} hidden rows, d={d}, V={V}, bf16 hidden states and head weight "
                    "(a 1B-class drafter's LM head at the Llama-3 vocabulary)",
        "ms_per_call": ms_f, "rows_per_s": R / (ms_f * 1e-3),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                     "frac": achieved / hbm_peak, "traffic": lmhead_traffic(),
                     "algorithmic_bytes_per_call": bytes_,
                     "kernel": "lmhead_tc_kernel (tcgen05 GEMM + statistics epilogue) and the row merge"},
        "tensor": {"achieved_tflops": tflops, "peak_tflops": tpeak, "frac": tflops / tpeak if tpeak else None,
                   "peak_source": "measured (MEASURED_PEAKS.json bf16_tflops, cuBLAS burst)" if tpeak else None,
                   "flops_per_call": flops},
        "unfused_ms": ms_u, "cublas_gemm_only_ms": ms_g, "speedup_vs_unfused": ms_u / ms_f,
        "parity": {"rows": int(len(rows)),
                   "argmax_equal": int(np.sum((g["argmax"][rows] == o["argmax"]) & clear)),
                   "argmax_compared": int(np.sum(clear)),
                   "max_abs_err": {k: float(np.max(np.abs(g[k][rows] - o[k]))) for k in ("H", "lse", "conf")},
                   "logit_rounding_bound": float(eps.max())},
        "timing": f"CUDA events over {calls} back-to-back calls after 5 warm-up calls; weight 525 MB > L2",
    }


def decode_sim_report(cmsd, torch, B=32, K=16, V=32000, iterations=512):
    """Algorithm 1 as a decode loop over device-generated f32 logits (k_next
    of each iteration is the next iteration's k_row), captured in a CUDA
    graph: the whole loop, generation alone, and the pass alone timed with
    CUDA events; then the ablation variants of Table III and the bonus row."""
    from paper_2508_15371_gb300 import decode_sim

    def one(preset="full", bonus=0, timing=False):
        p = cmsd.params(K, "sampled", preset=preset, bonus=bonus)
        sim = decode_sim.DecodeSim(B, K, V, iterations, p, seed=4)
        sim.step(0)                      # first launches outside the capture
        torch.cuda.synchronize()
        g = sim.capture()
        g.replay()
        torch.cuda.synchronize()
        hist = sim.history()
        s = decode_sim.summarize(hist, bonus=bool(bonus))
        if timing:
            gg = sim.capture(generate=True, verify=False)
            gv = sim.capture(generate=False, verify=True)
            e = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
            e[0].record()
            g.replay()
            e[1].record()
            gg.replay()
            e[2].record()
            gg.replay()
            e[3].record()
            gv.replay()
            e[4].record()
            gv.replay()
            e[5].record()
            torch.cuda.synchronize()
            ms, ms_gen, ms_pass = e[0].elapsed_time(e[1]), e[2].elapsed_time(e[3]), e[4].elapsed_time(e[5])
            hb = decode_sim.pass_bytes(hist, V, 4, bonus=bool(bonus))
            s.update({"ms_per_iteration": ms / iterations, "rows_per_s": s["rows"] / (ms * 1e-3),
                      "generation_ms_per_iteration": ms_gen / iterations,
                      "pass_ms_per_iteration": ms_pass / iterations,
                      "pass_rows_per_s": s["rows"] / (ms_pass * 1e-3),
                      "pass_bytes_per_iteration": hb / iterations,
                      "pass_gbs": hb / (ms_pass * 1e-3) / 1e9,
                      "timing": "CUDA graph of the 512 iterations; generation and pass also captured and "
                                "replayed alone (the pass over the last iteration's logits with the recorded "
                                "windows), CUDA events"})
        return s

    rep = one(timing=True)
    rep["workload"] = f"B={B} K_max={K} V={V} f32, {iterations} iterations, sampled rule, AR(1) spike heights"
    rep["ablation"] = {}
    keys = ("mean_k", "mean_accepted", "tokens_per_iteration", "rollbacks")
    for preset in ("full", "fixed_k", "fixed_tau", "fixed_k_tau", "entropy_only", "margin_only", "softmax_only"):
        s = one(preset)
        rep["ablation"][preset] = {k: s[k] for k in keys}
    s = one("full", bonus=1)
    rep["ablation"]["full+bonus_row"] = {k: s[k] for k in keys}
    return rep


# ---------------------------------------------------------------- our arm

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
    peak, peak_src = peaks()

    if args.only:
        # one workload's device-resident timing, nothing else (for profiling a
        # single configuration's launches)
        if args.only == "lmhead":
            print(json.dumps(lmhead_report(cmsd, torch, peak, calls=max(3, args.steps))), flush=True)
            return 0
        steps = max(3, args.steps)
        size = {"B": args.batch} if args.batch else {}
        print(json.dumps(bench_workload(cmsd, torch, dev, args.only, args.rule, steps, peak, **size)), flush=True)
        return 0

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

    # ---- timed region: device-resident inputs, two events ------------------
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    t_wall0 = time.time()
    ms_total = time_total(torch, calls, args.steps)
    t_wall1 = time.time()
    if dist:
        dist.barrier()
    # the same steps with an event after each: the spread of step times
    _, per_step = time_steps(torch, calls, args.steps)
    clocks.stop()
    clk = clocks.summary(t_wall0, t_wall1)
    # the same steps again with the library's per-kernel events (an event
    # between the two kernels serialises them, so this pass is not the one
    # `value` comes from): durations of the streaming and resample kernels
    k_ms, r_ms = kernel_times(cmsd, torch, calls, args.steps)
    n_last = out["n_accept"].cpu().numpy()
    rejected = int((n_last < K).sum()) if sampled else 0
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
    # two device input buffers: step j+1's inputs are copied (on a copy
    # stream) while step j computes; each step still copies all of its
    # inputs and reads its results back inside the timed region
    dbuf = [(torch.empty_like(host[0][0], device=dev), torch.empty_like(host[0][1], device=dev),
             torch.empty_like(host[0][2], device=dev)) for _ in range(2)]
    ecalls = [cmsd.FusedCall(db[0], db[1], db[2], p, seed=w0.seed, out=out, ws=ws) for db in dbuf]
    res_host = [torch.empty(B, dtype=torch.int32).pin_memory(), torch.empty((B, K), dtype=torch.int32).pin_memory(),
                torch.empty(B, dtype=torch.int32).pin_memory()]
    h2d = sum(x.numel() * x.element_size() for x in host[0])
    d2h = sum(x.numel() * x.element_size() for x in res_host)
    main = torch.cuda.current_stream()
    cs = torch.cuda.Stream()
    copied = [torch.cuda.Event() for _ in range(2)]
    computed = [torch.cuda.Event() for _ in range(2)]

    def e2e_steps_run(n, start_event=None):
        if start_event is not None:
            cs.wait_event(start_event)
        for j in range(n):
            hd, ht, hk = host[j % len(host)]
            db = dbuf[j % 2]
            with torch.cuda.stream(cs):
                if j >= 2:
                    cs.wait_event(computed[j % 2])     # the buffer's previous step is done
                db[0].copy_(hd, non_blocking=True)
                db[1].copy_(ht, non_blocking=True)
                db[2].copy_(hk, non_blocking=True)
                copied[j % 2].record(cs)
            main.wait_event(copied[j % 2])
            o = ecalls[j % 2](iteration=j)
            res_host[0].copy_(o["n_accept"], non_blocking=True)
            res_host[1].copy_(o["out_tokens"], non_blocking=True)
            res_host[2].copy_(o["k_next"], non_blocking=True)
            computed[j % 2].record(main)

    e2e_steps_run(3)
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    e2e_steps_run(e2e_steps, start_event=e0)
    e1.record()
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), dist, dev)
    e2e_value = job_rows_per_s(world, rows, e2e_steps, e2e_ms)
    del host, dbuf

    # ---- roofline: the streaming kernel, and the whole step -----------------
    k_med = statistics.median(k_ms)
    achieved = alg_bytes / (k_med * 1e-3) / 1e9
    step_stats = stats_ms(per_step)
    # the residual draw reads each rejected position's target row again (the
    # drafter groups it races are a few KB)
    resample_bytes = rejected * V * 2
    step_gbs = (alg_bytes + resample_bytes) / (ms_step * 1e-3) / 1e9

    if rank != 0:
        if dist:
            dist.destroy_process_group()
        return 0

    extra = {}
    if world == 1 and not args.no_extra:
        # ---- the other workloads ---------------------------------------------
        extra["workloads"] = [
            bench_workload(cmsd, torch, dev, "c1", "sampled", 200, peak, graph_latency=True),
            bench_workload(cmsd, torch, dev, "c1", "paper", 200, peak, graph_latency=True),
            bench_workload(cmsd, torch, dev, "c2", "sampled", 200, peak),
            bench_workload(cmsd, torch, dev, "c3", "paper", 200, peak, nsets=2),
            bench_workload(cmsd, torch, dev, "c4", "sampled", 50, peak),
            bench_workload(cmsd, torch, dev, "c4", "paper", 50, peak),
        ]
        # ---- decode-loop simulation --------------------------------------------
        if not args.no_decode_sim:
            extra["decode_sim"] = decode_sim_report(cmsd, torch)
        # ---- the drafter's LM head fused with the signals ----------------------
        extra["lmhead"] = lmhead_report(cmsd, torch, peak)

    # ---- CPU oracle baseline, with a live parity check of its sample ---------
    cpu = None
    if world == 1 and not args.no_cpu_baseline:
        it_live = 777
        gout = cmsd.confidence_verify(dsets[0][0], dsets[0][1], dsets[0][2], p=p, seed=w0.seed,
                                      iteration=it_live, signals=True)
        torch.cuda.synchronize()
        g = {k2: v2.cpu().numpy() for k2, v2 in gout.items() if v2 is not None}
        procs = max(1, min(16, host_cores()))
        v, nrows, dt, results = oracle_pool_run(w0, p.as_dict(), w0.seed, it_live, args.cpu_budget, procs)
        cpu = {"value": v, "unit": UNIT, "cores": procs, "kind": "oracle",
               "sample": f"{nrows} drafted positions ({nrows // K} whole sequences) of this workload, float64 "
                         f"numpy, {procs} worker processes (one per core), {dt:.1f} s"}
        extra["live_parity"] = live_parity(results, g, K)

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": C3_DESC, "rule": args.rule, "logits": "bf16", "accumulate": "f32",
                   "l2": "inputs larger than L2: 2 alternating input sets of 263 MB each (L2 129 MB)",
                   "parallelism": f"dp{world} (independent batches per GPU)" if world > 1 else "single GPU"},
        "step_ms": step_stats,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": ncu_traffic(WORKLOAD, args.rule),
                     "kernel": "stream_kernel (fused confidence + verify pass)",
                     "peak_source": f"{peak_src} (MEASURED_PEAKS.json hbm_gbs)" if peak_src == "measured"
                     else "fallback 6800 GB/s",
                     "algorithmic_bytes_per_launch": alg_bytes, "kernel_ms": k_med,
                     "kernel_timing": "CUDA events around each streaming-kernel launch (median over a second "
                                      "pass of the same steps)"},
        "step_roofline": {"achieved": step_gbs, "frac": step_gbs / peak, "unit": "GB/s",
                          "bytes_per_step": alg_bytes + resample_bytes,
                          "resample_bytes_per_step": resample_bytes,
                          "note": "every logit once plus the rejected positions' target rows again, over the "
                                  "median step"},
        "resample_ms": statistics.median(r_ms) if sampled else 0.0,
        "cpu_baseline": cpu,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "overlap": "step j+1's host-to-device copies run on a copy stream during step j's pass "
                           "(two device input buffers)",
                "steps": e2e_steps},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "parity": parity_record(WORKLOAD, args.rule),
        "outputs_written": "n_accept, out_tokens, k_next (the per-position signals H, margin, argmax, conf, "
                           "lse and the accept bits are not requested in the timed steps)",
    }
    line.update(extra)
    print(json.dumps(line), flush=True)
    if dist:
        dist.destroy_process_group()
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--rule", choices=["sampled", "paper"], default="sampled")
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle time for cpu_baseline")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-decode-sim", action="store_true", help="skip the decode-loop simulation report")
    ap.add_argument("--no-extra", action="store_true", help="headline only (no other workloads, no decode loop)")
    ap.add_argument("--only", choices=["c1", "c2", "c3", "c4", "lmhead"], default=None,
                    help="time one workload under --rule and print its object only (for profiling)")
    ap.add_argument("--batch", type=int, default=0, help="with --only: the number of sequences B (default: full)")
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
