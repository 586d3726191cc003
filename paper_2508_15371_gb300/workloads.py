"""Seeded synthetic inputs for the CM-ASD logits pass (numpy only).

This module generates logits, drafted tokens and decode-loop schedules; it
holds none of the method's arithmetic (no entropy, confidence, acceptance or
resampling).  It is the one module that serves both the CUDA path (tests and
bench.py feed its arrays to the library) and the CPU oracle (tests hand it the
same arrays).

The paper's workloads are WMT / CNN-DailyMail logits from trained drafter and
verifier models (Sec. IV.A); those are not available, so these recipes stand
in for them with the vocabulary sizes of encoder-decoder MT/summarisation
models (32000, 32128) and of LLM heads (128256, 152064), and with spike
heights, noise levels and mixtures chosen to span peaked to flat
distributions.

Recipes (rows = B*K drafted positions, each with a V-long drafter and target
logit row; float32 values, rounded to bfloat16 with round-to-nearest-even for
the bf16 recipes):

  c1  f32.  z = N(0,1) + spike U[0,12] on a uniform token; target =
      z + 0.5 N(0,1); drafted token = argmax z.
  c2  bf16. z = 1.5 N(0,1) + spike U[0,10]; target = z + sigma_b N(0,1),
      sigma_b cycling over (0.2, 1.0, 3.0) by sequence; drafted tokens sampled
      from softmax(z) (Gumbel-max on the rounded logits).
  c3  bf16. Zipf-shaped profile over a per-row random permutation of the
      vocabulary, scaled by 4, plus 0.5 N(0,1); target = z + N(0,1); drafted
      tokens sampled.  profile="rank": z = 4 r^-1.1 (rank weights used as
      logits); profile="log": z = -4 * 1.1 * ln r (a Zipf probability law).
  c4  bf16. Per row: 50% peaked (N(0,1) + spike U[8,14]), 30% flat
      (0.3 N(0,1)), 20% bimodal (N(0,1) + spikes h and h - U[0,0.5],
      h ~ U[8,14]); target = z + 2 N(0,1); drafted tokens sampled.
  c5  f32 decode-loop simulation, generated per iteration from Philox
      (see decode_iteration_host); bit-identical to the device generator in
      libcmsd_workload.so.

Rows are generated in fixed blocks of ROW_BLOCK rows, block j from child j of
numpy's SeedSequence(seed), so results do not depend on thread count.
"""
from __future__ import annotations

import concurrent.futures as _cf
import os
from dataclasses import dataclass

import numpy as np

ROW_BLOCK = 16

FULL_SIZES = {
    "c1": dict(B=1, K=4, V=32000, dtype="f32", seed=0),
    "c2": dict(B=8, K=8, V=32128, dtype="bf16", seed=1),
    "c3": dict(B=64, K=8, V=128256, dtype="bf16", seed=2),
    "c4": dict(B=256, K=16, V=152064, dtype="bf16", seed=3),
    "c5": dict(B=32, K=16, V=32000, dtype="f32", seed=4, iterations=512),
}


@dataclass
class Workload:
    name: str
    B: int
    K: int
    V: int
    dtype: str            # "f32" (float32 arrays) or "bf16" (uint16 bit patterns)
    draft: np.ndarray     # [B, K, V]
    target: np.ndarray    # [B, K, V]
    tokens: np.ndarray    # int32 [B, K]
    seed: int             # Philox seed for the method's uniforms
    k_row: np.ndarray = None
    note: str = ""

    @property
    def rows(self):
        return self.B * self.K

    @property
    def logit_bytes(self):
        es = 4 if self.dtype == "f32" else 2
        return 2 * self.B * self.K * self.V * es


# ---------------------------------------------------------------------------
# bfloat16 rounding (round to nearest even), numpy only
# ---------------------------------------------------------------------------

def f32_to_bf16_bits(x):
    """float32 -> bfloat16 bit patterns (uint16), round-to-nearest-even.

    Infinities are preserved; NaN is not expected in these recipes.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits):
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32)


# ---------------------------------------------------------------------------
# blockwise generation helpers
# ---------------------------------------------------------------------------

def _blocks(nrows):
    return [(r0, min(nrows, r0 + ROW_BLOCK)) for r0 in range(0, nrows, ROW_BLOCK)]


def _run_blocks(seed, nrows, fn, threads=None):
    blocks = _blocks(nrows)
    children = np.random.SeedSequence(seed).spawn(len(blocks))
    jobs = [(np.random.Generator(np.random.PCG64(c)), r0, r1) for c, (r0, r1) in zip(children, blocks)]
    if threads is None:
        threads = min(16, os.cpu_count() or 1)
    if threads <= 1 or len(jobs) == 1:
        for g, r0, r1 in jobs:
            fn(g, r0, r1)
        return
    with _cf.ThreadPoolExecutor(threads) as ex:
        list(ex.map(lambda j: fn(*j), jobs))


def _gumbel_sample(rng, z32):
    """Drafted tokens sampled from softmax(z) (the drafter's own sampling)."""
    u = rng.random(z32.shape)
    g = -np.log(-np.log(u))
    return np.argmax(z32.astype(np.float64) + g, axis=-1)


def _finish(name, B, K, V, dtype, seed, d32, t32, tokens, note):
    if dtype == "bf16":
        draft = f32_to_bf16_bits(d32).reshape(B, K, V)
        target = f32_to_bf16_bits(t32).reshape(B, K, V)
    else:
        draft = d32.reshape(B, K, V)
        target = t32.reshape(B, K, V)
    return Workload(name=name, B=B, K=K, V=V, dtype=dtype, draft=draft, target=target,
                    tokens=tokens.reshape(B, K).astype(np.int32), seed=seed, note=note)


# ---------------------------------------------------------------------------
# recipes c1 - c4
# ---------------------------------------------------------------------------

def make_c1(B=1, K=4, V=32000, seed=0, dtype="f32", threads=None):
    n = B * K
    d = np.empty((n, V), np.float32)
    t = np.empty((n, V), np.float32)
    tok = np.empty(n, np.int64)

    def blk(g, r0, r1):
        m = r1 - r0
        z = g.standard_normal((m, V), dtype=np.float32)
        spike = g.integers(0, V, m)
        h = g.uniform(0.0, 12.0, m).astype(np.float32)
        z[np.arange(m), spike] += h
        d[r0:r1] = z
        t[r0:r1] = z + np.float32(0.5) * g.standard_normal((m, V), dtype=np.float32)
        zr = z if dtype == "f32" else bf16_bits_to_f32(f32_to_bf16_bits(z))
        tok[r0:r1] = np.argmax(zr, axis=-1)

    _run_blocks(seed, n, blk, threads)
    return _finish("c1", B, K, V, dtype, seed, d, t, tok,
                   "N(0,1)+spike U[0,12]; target +0.5N; drafted = argmax")


def make_c2(B=8, K=8, V=32128, seed=1, dtype="bf16", threads=None):
    n = B * K
    d = np.empty((n, V), np.float32)
    t = np.empty((n, V), np.float32)
    tok = np.empty(n, np.int64)
    sig = np.array([0.2, 1.0, 3.0], np.float32)

    def blk(g, r0, r1):
        m = r1 - r0
        z = np.float32(1.5) * g.standard_normal((m, V), dtype=np.float32)
        spike = g.integers(0, V, m)
        h = g.uniform(0.0, 10.0, m).astype(np.float32)
        z[np.arange(m), spike] += h
        s = sig[(np.arange(r0, r1) // K) % 3][:, None]
        d[r0:r1] = z
        t[r0:r1] = z + s * g.standard_normal((m, V), dtype=np.float32)
        zr = z if dtype == "f32" else bf16_bits_to_f32(f32_to_bf16_bits(z))
        tok[r0:r1] = _gumbel_sample(g, zr)

    _run_blocks(seed, n, blk, threads)
    return _finish("c2", B, K, V, dtype, seed, d, t, tok,
                   "1.5N+spike U[0,10]; target +sigma_b N, sigma cycles 0.2/1/3; drafted ~ softmax")


def zipf_profile(V, kind="rank"):
    r = np.arange(1, V + 1, dtype=np.float64)
    if kind == "rank":
        return (4.0 * r ** -1.1).astype(np.float32)
    if kind == "log":
        return (-4.0 * 1.1 * np.log(r)).astype(np.float32)
    raise ValueError(kind)


def make_c3(B=64, K=8, V=128256, seed=2, dtype="bf16", profile="rank", threads=None):
    n = B * K
    d = np.empty((n, V), np.float32)
    t = np.empty((n, V), np.float32)
    tok = np.empty(n, np.int64)
    prof = zipf_profile(V, profile)

    def blk(g, r0, r1):
        m = r1 - r0
        perm = g.permuted(np.tile(np.arange(V), (m, 1)), axis=1)
        z = prof[perm] + np.float32(0.5) * g.standard_normal((m, V), dtype=np.float32)
        d[r0:r1] = z
        t[r0:r1] = z + g.standard_normal((m, V), dtype=np.float32)
        zr = z if dtype == "f32" else bf16_bits_to_f32(f32_to_bf16_bits(z))
        tok[r0:r1] = _gumbel_sample(g, zr)

    _run_blocks(seed, n, blk, threads)
    return _finish("c3", B, K, V, dtype, seed, d, t, tok,
                   f"4x Zipf(1.1) profile ({profile}) over a per-row permutation +0.5N; "
                   "target +N; drafted ~ softmax")


def make_c4(B=256, K=16, V=152064, seed=3, dtype="bf16", threads=None):
    n = B * K
    d = np.empty((n, V), np.float32)
    t = np.empty((n, V), np.float32)
    tok = np.empty(n, np.int64)

    def blk(g, r0, r1):
        m = r1 - r0
        kind = g.choice(3, size=m, p=[0.5, 0.3, 0.2])
        z = g.standard_normal((m, V), dtype=np.float32)
        flat = kind == 1
        z[flat] *= np.float32(0.3)
        h = g.uniform(8.0, 14.0, m).astype(np.float32)
        t1 = g.integers(0, V, m)
        t2 = (t1 + 1 + g.integers(0, V - 1, m)) % V
        dh = g.uniform(0.0, 0.5, m).astype(np.float32)
        rows = np.arange(m)
        peak = kind != 1
        z[rows[peak], t1[peak]] += h[peak]
        bi = kind == 2
        z[rows[bi], t2[bi]] += h[bi] - dh[bi]
        d[r0:r1] = z
        t[r0:r1] = z + np.float32(2.0) * g.standard_normal((m, V), dtype=np.float32)
        zr = z if dtype == "f32" else bf16_bits_to_f32(f32_to_bf16_bits(z))
        tok[r0:r1] = _gumbel_sample(g, zr)

    _run_blocks(seed, n, blk, threads)
    return _finish("c4", B, K, V, dtype, seed, d, t, tok,
                   "mixture 50% peaked U[8,14] / 30% flat 0.3N / 20% bimodal; target +2N; drafted ~ softmax")


RECIPES = {"c1": make_c1, "c2": make_c2, "c3": make_c3, "c4": make_c4}


# ---------------------------------------------------------------------------
# drafter LM head: hidden states and weights (the fused LM-head entry point)
# ---------------------------------------------------------------------------

@dataclass
class LMHeadWorkload:
    name: str
    R: int
    d: int
    V: int
    seed: int
    hidden: np.ndarray      # uint16 bf16 bits [R, d]
    weight: np.ndarray      # uint16 bf16 bits [V, d]
    spike_token: np.ndarray  # int64 [R]: the vocabulary row a hidden state points at (-1: none)
    note: str


def make_lmhead(R=64, d=2048, V=128256, seed=5, exact=False, spiked=0.7):
    """Hidden states [R, d] and an LM-head weight [V, d], bf16, seeded.

    Default recipe (a 1B-class drafter's head at a Llama-3-sized vocabulary):
    W[v, j] ~ N(0, 1) / sqrt(d); each hidden state is N(0, 0.7^2) noise, and
    with probability `spiked` also points at a uniform vocabulary row v* with
    a height a ~ U[0, 20] (h += a W[v*] / |W[v*]|^2), so the logit at v* is
    raised by about a: a spread from flat to peaked rows (at V = 128256 the
    noise logits alone have a maximum near 3 and a sum near 1.6e5, so a
    spike needs a height of about 12 to hold half the probability).

    exact=True: every entry is a multiple of 1/16 (W in [-1/8, 1/8], h in
    [-1/4, 1/4], a spiked row adds W[v*]), so each product is a multiple of
    2^-8 and every partial sum of a dot product is exact in float32 for
    d <= 2^14: float32 logits then equal the float64 ones in any order.
    """
    rng = np.random.default_rng(np.random.SeedSequence([seed, R, d, V, int(exact)]))
    if exact:
        w32 = rng.integers(-2, 3, size=(V, d), dtype=np.int8).astype(np.float32) / np.float32(16.0)
        h32 = rng.integers(-2, 3, size=(R, d), dtype=np.int8).astype(np.float32) / np.float32(16.0)
    else:
        w32 = (rng.standard_normal((V, d), dtype=np.float32) / np.float32(np.sqrt(d))).astype(np.float32)
        h32 = (0.7 * rng.standard_normal((R, d), dtype=np.float32)).astype(np.float32)
    wb = f32_to_bf16_bits(w32)
    wq = bf16_bits_to_f32(wb)
    spike = np.full(R, -1, dtype=np.int64)
    for r in range(R):
        if rng.random() < spiked:
            v = int(rng.integers(0, V))
            spike[r] = v
            if exact:
                h32[r] += wq[v]
            else:
                a = rng.uniform(0.0, 20.0)
                h32[r] += np.float32(a) * wq[v] / np.float32(np.dot(wq[v], wq[v]))
    hb = f32_to_bf16_bits(h32)
    note = ("entries are multiples of 1/16 (float32 dot products exact)" if exact else
            "W ~ N(0,1)/sqrt(d); h ~ N(0,0.7^2) plus a spike of height U[0,20] towards a uniform token "
            "on %.0f%% of rows" % (100 * spiked))
    return LMHeadWorkload("lmhead", R, d, V, seed, hb, wb, spike, note)


def make(name, **kw):
    """Full-size recipe `name`, with any size/seed overridden by keyword."""
    base = dict(FULL_SIZES[name])
    base.pop("iterations", None)
    base.update(kw)
    return RECIPES[name](**base)


# ---------------------------------------------------------------------------
# c5: decode-loop simulation inputs, bit-identical on host and device
# ---------------------------------------------------------------------------

MASK32 = 0xFFFFFFFF
_PH_M0, _PH_M1 = 0xD2511F53, 0xCD9E8D57
_PH_W0, _PH_W1 = 0x9E3779B9, 0xBB67AE85

# Philox counter word 3 for the generator's streams (kept away from the
# method's own (iteration << 2 | purpose) values).
GEN_DNOISE = 0xC0000002
GEN_TNOISE = 0xC0000003
GEN_SPIKE = 0xC0000004
GEN_AR = 0xC0000005

C5_RHO = 0.9
C5_MU = 6.0
C5_SIGMA = 1.5
C5_TARGET_NOISE = 0.8
C5_HMAX = 12.0


def _philox_np(c0, c1, c2, c3, k0, k1):
    """Philox4x32-10 over uint64 arrays (generator copy; see Salmon et al. 2011)."""
    c0, c1, c2, c3 = np.broadcast_arrays(*(np.asarray(c, dtype=np.uint64) & np.uint64(MASK32)
                                           for c in (c0, c1, c2, c3)))
    k0, k1 = int(k0) & MASK32, int(k1) & MASK32
    mask, s32 = np.uint64(MASK32), np.uint64(32)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + _PH_W0) & MASK32
            k1 = (k1 + _PH_W1) & MASK32
        p0 = np.uint64(_PH_M0) * c0
        p1 = np.uint64(_PH_M1) * c2
        c0, c1, c2, c3 = (((p1 >> s32) ^ c1 ^ np.uint64(k0)) & mask, p1 & mask,
                          ((p0 >> s32) ^ c3 ^ np.uint64(k1)) & mask, p0 & mask)
    return c0, c1, c2, c3


NORMAL_BITS = 13          # the table's size: 2**13 float32 (32 KB, held in shared memory on the device)


def normal_table(bits=NORMAL_BITS):
    """Quantiles of N(0,1) at the midpoints (k + 1/2) / 2**bits, as float32.

    The top `bits` bits of a 16-bit uniform index it, giving a discretised
    normal that host and device reproduce exactly (a table lookup, no
    transcendental calls).
    """
    from scipy.special import ndtri
    n = 1 << bits
    return ndtri((np.arange(n, dtype=np.float64) + 0.5) / n).astype(np.float32)


def _u16_stream(seed, row, it, purpose, V):
    """16-bit uniforms for v = 0..V-1: counter (v >> 3, row, it, purpose),
    word (v >> 1) & 3, low half for even v, high half for odd v."""
    ngrp = (V + 7) // 8
    w = _philox_np(np.arange(ngrp, dtype=np.uint64), row, it, purpose, seed & MASK32, seed >> 32)
    words = np.stack(w, axis=1).reshape(-1)                        # 4 words per group
    halves = np.stack([words & np.uint64(0xFFFF), words >> np.uint64(16)], axis=1).reshape(-1)
    return halves[:V].astype(np.int64)


def ar1_heights(B, iterations, seed=4, table=None):
    """Per-sequence spike heights h[it, b] of the c5 drafter rows (float32).

    h_{-1} = mu; h_it = clip((rho * h_{it-1} + (1 - rho) * mu) + sigma * eps, 0, 12)
    with eps from the normal table; every operation rounded to float32 in this
    order (the device generator reads this table, it does not recompute it).
    """
    if table is None:
        table = normal_table()
    rho = np.float32(C5_RHO)
    c = np.float32(np.float32(1.0) - rho) * np.float32(C5_MU)
    sg = np.float32(C5_SIGMA)
    h = np.full(B, np.float32(C5_MU), np.float32)
    out = np.empty((iterations, B), np.float32)
    b = np.arange(B, dtype=np.uint64)
    for it in range(iterations):
        w0, _, _, _ = _philox_np(np.uint64(0), b, it, GEN_AR, seed & MASK32, seed >> 32)
        eps = table[((w0 & np.uint64(0xFFFF)) >> np.uint64(16 - NORMAL_BITS)).astype(np.int64)]
        h = (rho * h + c) + sg * eps
        h = np.minimum(np.float32(C5_HMAX), np.maximum(np.float32(0.0), h)).astype(np.float32)
        out[it] = h
    return out


def decode_row_host(table, heights, it, b, i, K_max, V, seed=4):
    """One c5 row (b, i) at iteration it: (drafter f32[V], target f32[V], drafted token).

    Generator row id b * (K_max + 1) + i (room for the verifier's extra row at
    i = K_max).  drafter z = n1 + h[it, b] at the spike token; target = z +
    0.8 * n2 (float32, multiply then add); drafted token = first argmax of z.
    """
    row = b * (K_max + 1) + i
    n1 = table[_u16_stream(seed, row, it, GEN_DNOISE, V) >> (16 - NORMAL_BITS)]
    n2 = table[_u16_stream(seed, row, it, GEN_TNOISE, V) >> (16 - NORMAL_BITS)]
    w0, _, _, _ = _philox_np(np.uint64(0), row, it, GEN_SPIKE, seed & MASK32, seed >> 32)
    tok = int((int(w0) * V) >> 32)
    z = n1.copy()
    z[tok] = np.float32(z[tok] + heights[it, b])
    tgt = (z + np.float32(C5_TARGET_NOISE) * n2).astype(np.float32)
    return z, tgt, int(np.argmax(z))


def decode_iteration_host(table, heights, it, b, k, K_max, V, seed=4, bonus=False):
    """Rows i < k of sequence b at iteration it: drafter [k, V], target
    [k, V] (or [k + 1, V] with the verifier's extra row) and tokens [k]."""
    kt = k + 1 if bonus else k
    d = np.empty((k, V), np.float32)
    t = np.empty((kt, V), np.float32)
    tok = np.empty(k, np.int64)
    for i in range(kt):
        di, ti, ki = decode_row_host(table, heights, it, b, i, K_max, V, seed)
        t[i] = ti
        if i < k:
            d[i], tok[i] = di, ki
    return d, t, tok
