"""Philox4x32-10 counter-based generator for the oracle (test infrastructure).

Written from the published definition (Salmon, Moraes, Dror, Shaw,
"Parallel Random Numbers: As Easy as 1, 2, 3", SC'11): a 4 x 32-bit counter
is passed through ten rounds; each round multiplies counter words 0 and 2 by
fixed odd constants, swaps the high/low halves into a new word order and
XORs in the key, and the 2 x 32-bit key is advanced by two Weyl constants
between rounds.

The paper being restated (arXiv 2508.15371) does not say how its random
draws are made; the speculative-sampling acceptance it cites (Sec. II, [5],
[6]) only needs uniforms.  This module fixes the reading used on both sides of
the parity test: key = (seed low word, seed high word), counter layout

    acceptance  u  : counter (0,      b, i, (iteration << 2) | 0), word 0
    residual    U_v: counter (v >> 2, b, n, (iteration << 2) | 1), word v & 3
    residual    U_g: counter (g >> 2, b, n, (iteration << 2) | 2), word g & 3
                     (one draw per group g of GROUP = 32 vocabulary entries)

and a 24-bit uniform u = (word >> 8) * 2**-24 in [0, 1), exact in float32.

Nothing here is shared with the CUDA library; the pin for this code is
tests/test_philox_pin.py (an independent Philox implementation).
"""
from __future__ import annotations

import numpy as np

MASK32 = 0xFFFFFFFF
# Round multipliers and Weyl key increments of Philox4x32 (Salmon et al. 2011).
PHILOX_M0 = 0xD2511F53
PHILOX_M1 = 0xCD9E8D57
PHILOX_W0 = 0x9E3779B9
PHILOX_W1 = 0xBB67AE85
ROUNDS = 10

PURPOSE_ACCEPT = 0
PURPOSE_RESIDUAL = 1
PURPOSE_GROUP = 2
GROUP = 32


def philox4x32_10(counter, key):
    """One Philox4x32-10 block: 4 counter words, 2 key words -> 4 output words.

    Pure Python integers; slow but transparent.
    """
    c0, c1, c2, c3 = (int(x) & MASK32 for x in counter)
    k0, k1 = (int(x) & MASK32 for x in key)
    for rnd in range(ROUNDS):
        if rnd:
            k0 = (k0 + PHILOX_W0) & MASK32
            k1 = (k1 + PHILOX_W1) & MASK32
        p0 = PHILOX_M0 * c0
        p1 = PHILOX_M1 * c2
        c0, c1, c2, c3 = (
            ((p1 >> 32) ^ c1 ^ k0) & MASK32,
            p1 & MASK32,
            ((p0 >> 32) ^ c3 ^ k1) & MASK32,
            p0 & MASK32,
        )
    return (c0, c1, c2, c3)


def philox4x32_10_np(c0, c1, c2, c3, k0, k1):
    """Vectorised Philox4x32-10 over numpy arrays of counters (broadcasting).

    Products of two 32-bit words are formed exactly in uint64.
    Returns four uint32 arrays.
    """
    c0 = np.asarray(c0, dtype=np.uint64) & MASK32
    c1 = np.asarray(c1, dtype=np.uint64) & MASK32
    c2 = np.asarray(c2, dtype=np.uint64) & MASK32
    c3 = np.asarray(c3, dtype=np.uint64) & MASK32
    c0, c1, c2, c3 = np.broadcast_arrays(c0, c1, c2, c3)
    k0 = np.uint64(int(k0) & MASK32)
    k1 = np.uint64(int(k1) & MASK32)
    m0 = np.uint64(PHILOX_M0)
    m1 = np.uint64(PHILOX_M1)
    mask = np.uint64(MASK32)
    s32 = np.uint64(32)
    for rnd in range(ROUNDS):
        if rnd:
            k0 = np.uint64((int(k0) + PHILOX_W0) & MASK32)
            k1 = np.uint64((int(k1) + PHILOX_W1) & MASK32)
        p0 = m0 * c0
        p1 = m1 * c2
        c0, c1, c2, c3 = (
            ((p1 >> s32) ^ c1 ^ k0) & mask,
            p1 & mask,
            ((p0 >> s32) ^ c3 ^ k1) & mask,
            p0 & mask,
        )
    return (c0.astype(np.uint32), c1.astype(np.uint32),
            c2.astype(np.uint32), c3.astype(np.uint32))


def seed_key(seed):
    seed = int(seed) & 0xFFFFFFFFFFFFFFFF
    return (seed & MASK32, seed >> 32)


def word_to_unit(word):
    """24-bit uniform in [0, 1): (word >> 8) * 2**-24 (exact in float32 and float64)."""
    if isinstance(word, np.ndarray):
        return (word >> np.uint32(8)).astype(np.float64) * (2.0 ** -24)
    return (int(word) >> 8) * (2.0 ** -24)


def accept_uniform(seed, b, i, iteration):
    """Uniform u for the acceptance test of drafted position i of sequence b."""
    ctr = (0, b, i, ((int(iteration) << 2) | PURPOSE_ACCEPT) & MASK32)
    return word_to_unit(philox4x32_10(ctr, seed_key(seed))[0])


def residual_uniforms(seed, b, n, iteration, V):
    """Uniforms U_v, v = 0..V-1, for the residual draw at position n of sequence b."""
    k0, k1 = seed_key(seed)
    ngrp = (V + 3) // 4
    grp = np.arange(ngrp, dtype=np.uint64)
    c3 = ((int(iteration) << 2) | PURPOSE_RESIDUAL) & MASK32
    w = philox4x32_10_np(grp, b, n, c3, k0, k1)
    words = np.stack(w, axis=1).reshape(-1)[:V]
    return word_to_unit(words)


def group_uniforms(seed, b, n, iteration, ngroups):
    """Uniforms U_g, g = 0..ngroups-1, of the group-level residual draw."""
    k0, k1 = seed_key(seed)
    nblk = (ngroups + 3) // 4
    blk = np.arange(nblk, dtype=np.uint64)
    c3 = ((int(iteration) << 2) | PURPOSE_GROUP) & MASK32
    w = philox4x32_10_np(blk, b, n, c3, k0, k1)
    words = np.stack(w, axis=1).reshape(-1)[:ngroups]
    return word_to_unit(words)
