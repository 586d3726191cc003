"""The CPU oracle over many sequences at once, in a pool of worker processes.

Test infrastructure: the full-size parity tests compare every sequence of a
workload with the oracle, which takes minutes on one core (about 300 rows/s at
V = 128256).  Sequences are independent, so they are split over the host's
cores.  The pool is started with the `spawn` method, so that no worker is a
fork of a process that already holds a CUDA context.

Each worker runs the oracle's own public functions on a slice of sequences
and returns plain arrays; nothing here computes any part of the method.
"""
from __future__ import annotations

import atexit
import multiprocessing as mp
import os
from types import SimpleNamespace

import numpy as np

_pool = None


def nproc():
    try:
        n = len(os.sched_getaffinity(0))
    except AttributeError:   # pragma: no cover
        n = os.cpu_count() or 1
    return max(1, min(16, n))


def pool():
    """The shared spawn-context pool (created on first use)."""
    global _pool
    if _pool is None:
        _pool = mp.get_context("spawn").Pool(nproc())
        atexit.register(close)
    return _pool


def close():
    global _pool
    if _pool is not None:
        _pool.terminate()
        _pool.join()
        _pool = None


# ------------------------------------------------------------------ workers

def _fused_task(task):
    """Oracle over one slice of sequences (global indices b_index)."""
    draft, target, tokens, dtype, pdict, seed, iteration, k_rows, b_index = task
    import oracle as O
    P = O.Params(**pdict)
    out = []
    for j, b in enumerate(b_index):
        kb = int(k_rows[j])
        d = O.logits_to_f64(draft[j:j + 1], dtype)
        t = O.logits_to_f64(target[j:j + 1], dtype)
        r = O.confidence(d, P, k_row=[kb])
        v = O.verify_sequence(d[0], t[0], tokens[j], r.conf[0], kb, P, seed, int(b), iteration)
        out.append(dict(b=int(b), H=r.H[0], margin=r.margin[0], psm=r.psm[0], argmax=r.argmax[0],
                        conf=r.conf[0], lse=r.lse[0], k_next=int(r.k_next[0]), k_flag=bool(r.k_flag[0]),
                        **v))
    return out


def _decode_task(task):
    """Oracle replay of one decode-loop sequence (Algorithm 1 over the c5 rows)."""
    b, B, K, V, iterations, pdict, seed = task
    import oracle as O
    from paper_2508_15371_gb300 import workloads as W
    table = W.normal_table()
    heights = W.ar1_heights(B, iterations, seed, table)

    def gen(it, bb, k):
        return W.decode_iteration_host(table, heights, it, bb, k, K, V, seed, bonus=bool(pdict.get("bonus")))

    return b, O.decode_sim_sequence(gen, b, iterations, K, O.Params(**pdict), seed)


# ------------------------------------------------------------------ drivers

def fused(w, pdict, seed, iteration=0, k_row=None, seqs=None, chunk=None):
    """oracle.confidence_verify over the sequences `seqs` of workload w (all
    by default), in the pool.  Returns a namespace with the same [B, K] / [B]
    arrays as oracle.Result (NaN / -1 where a sequence was not evaluated)."""
    B, K, V = w.B, w.K, w.V
    kb = np.full(B, K, np.int64) if k_row is None else np.asarray(k_row, np.int64)
    seq_list = list(range(B)) if seqs is None else [int(b) for b in seqs]
    if chunk is None:
        chunk = max(1, len(seq_list) // (4 * nproc()))
    tasks = []
    for s0 in range(0, len(seq_list), chunk):
        bs = seq_list[s0:s0 + chunk]
        tasks.append((np.ascontiguousarray(w.draft[bs]), np.ascontiguousarray(w.target[bs]),
                      np.ascontiguousarray(w.tokens[bs]), w.dtype, dict(pdict), seed, iteration, kb[bs],
                      bs))
    Kout = K + 1 if pdict.get("bonus") else K
    r = SimpleNamespace(
        H=np.full((B, K), np.nan), margin=np.full((B, K), np.nan), psm=np.full((B, K), np.nan),
        conf=np.full((B, K), np.nan), lse=np.full((B, K), np.nan), argmax=np.full((B, K), -1, np.int64),
        k_next=np.full(B, -1, np.int64), k_flag=np.zeros(B, bool), accept=np.zeros((B, K), bool),
        acc_flag=np.zeros((B, K), bool), n_accept=np.full(B, -1, np.int64), n_flag=np.zeros(B, bool),
        out_tokens=np.full((B, Kout), -1, np.int64), tok_flag=np.zeros(B, bool),
        target_argmax=np.full((B, K), -1, np.int64))
    for part in pool().imap_unordered(_fused_task, tasks):
        for s in part:
            b, k = s["b"], int(kb[s["b"]])
            for n in ("H", "margin", "psm", "conf", "lse", "argmax"):
                getattr(r, n)[b] = s[n]
            r.k_next[b], r.k_flag[b] = s["k_next"], s["k_flag"]
            r.accept[b, :k], r.acc_flag[b, :k] = s["accept"], s["acc_flag"]
            r.n_accept[b], r.n_flag[b] = s["n_accept"], s["n_flag"]
            r.out_tokens[b], r.tok_flag[b] = s["out_tokens"], s["tok_flag"]
            r.target_argmax[b, :k] = s["target_argmax"]
    return r


def decode_replays(B, K, V, iterations, pdict, seed, seqs):
    """{b: oracle.decode_sim_sequence trajectory} for the sequences seqs."""
    tasks = [(int(b), B, K, V, iterations, dict(pdict), seed) for b in seqs]
    return dict(pool().imap_unordered(_decode_task, tasks))
