"""The arithmetic claims behind the residual draw by group bounds, checked in
float32 on the CPU (no GPU, no oracle).

The draw skips a group g when U_g f > K1 Rb_g (f = 0.99999), where K1 is the
exact key of some group, and
  Rb_g = fl(fl(p(m_g)) (32 + 1/2048)) + 2^-100,   m_g the group's largest target logit,
  p(z) = fl(fl(2^fl(z log2e - M log2e)) / S).
It is sound if every skipped group's computed key fl(E_g / R_g) exceeds K1, with
  R_g = the float32 sum of max(0, p_v - q_v) over the group's 32 entries,
  E_g = -log1p(-U_g).
Two claims carry this, and both are checked here under float32 rounding:
  1. R_g <= Rb_g, even when each 2^x carries a relative error of up to 2^-21
     (the budget allowed for the hardware's ex2) chosen against the bound;
  2. U_g f > K1 Rb_g implies fl(E_g / R_g) > K1, for K1 placed just below,
     at and above each group's bound U_g / Rb_g.
"""
import numpy as np
import pytest

F32 = np.float32
LOG2E = F32(1.4426950408889634)
SCALE = F32(32.0 + 1.0 / 2048.0)
FLOOR = F32(2.0 ** -100)
FILTER = F32(0.99999)
EX2_ERR = 2.0 ** -21


def _p(z, ml, inv_s, err):
    """p = fl(fl(2^fl(z log2e - ml)) inv_s), with 2^x scaled by (1 + err)."""
    x = (z * LOG2E - ml).astype(F32)
    e = np.exp2(x.astype(np.float64)) * (1.0 + err)
    return (e.astype(F32) * inv_s).astype(F32)


def _group_sum(r):
    """The float32 sum of 32 entries in the kernel's order: pairs of 8-entry
    lanes summed in packed halves, then the four lanes by xor shuffles."""
    lanes = r.reshape(4, 8)
    lo = np.zeros(4, F32)
    hi = np.zeros(4, F32)
    for k in range(4):
        lo = (lo + lanes[:, 2 * k]).astype(F32)
        hi = (hi + lanes[:, 2 * k + 1]).astype(F32)
    acc = (lo + hi).astype(F32)
    for o in (1, 2):
        acc = (acc + acc[np.arange(4) ^ o]).astype(F32)
    return acc[0]


def _rows(rng, n):
    for _ in range(n):
        kind = rng.integers(5)
        if kind == 0:      # peaked
            zt = rng.normal(0, 1, 32 * 64).astype(F32)
            zt[rng.integers(zt.size)] += F32(rng.uniform(5, 15))
        elif kind == 1:    # flat
            zt = rng.normal(0, 0.02, 32 * 64).astype(F32)
        elif kind == 2:    # a wide spread, many p near underflow
            zt = rng.normal(0, 30, 32 * 64).astype(F32)
        elif kind == 3:    # groups that repeat their maximum
            zt = rng.normal(0, 2, 32 * 64).astype(F32)
            zt.reshape(64, 32)[:, 1] = zt.reshape(64, 32).max(axis=1)
        else:              # groups of 32 equal logits and no drafter mass past entry 0: the bound at its tightest
            zt = np.repeat(rng.normal(0, 1, 64).astype(F32), 32)
            zd = np.full(zt.size, -1e4, F32)
            zd[0] = 0
            yield zt, zd
            continue
        zd = (zt + rng.normal(0, 1, zt.size)).astype(F32)
        yield zt, zd


@pytest.fixture(autouse=True)
def _quiet():
    with np.errstate(over="ignore", divide="ignore", invalid="ignore"):
        yield


def test_group_mass_below_its_bound():
    rng = np.random.default_rng(0)
    checked = 0
    for zt, zd in _rows(rng, 60):
        M = zt.max()
        ml = (M * LOG2E).astype(F32)
        S = np.exp(zt.astype(np.float64) - float(M)).sum()
        inv_s = F32(1.0 / S)
        md = zd.max()
        ninv_sd = F32(-1.0 / np.exp(zd.astype(np.float64) - float(md)).sum())
        mld = (md * LOG2E).astype(F32)
        for g in range(zt.size // 32):
            zg, dg = zt[32 * g: 32 * g + 32], zd[32 * g: 32 * g + 32]
            m = zg.max()
            # the bound's 2^x as small as the budget allows, the entries' as large
            pm = _p(np.array([m], F32), ml, inv_s, -EX2_ERR)[0]
            rb = F32(F32(pm * SCALE) + FLOOR)
            p = _p(zg, ml, inv_s, +EX2_ERR)
            qn = _p(dg, mld, ninv_sd, 0.0)          # -q, rounded the same way
            r = np.maximum((p + qn).astype(F32), F32(0))
            acc = _group_sum(r)
            assert acc <= rb, (g, float(acc), float(rb))
            checked += 1
    assert checked == 60 * 64


def test_skipped_groups_cannot_win_or_tie():
    rng = np.random.default_rng(1)
    skipped = 0
    for zt, zd in _rows(rng, 40):
        M = zt.max()
        ml = (M * LOG2E).astype(F32)
        inv_s = F32(1.0 / np.exp(zt.astype(np.float64) - float(M)).sum())
        md = zd.max()
        mld = (md * LOG2E).astype(F32)
        ninv_sd = F32(-1.0 / np.exp(zd.astype(np.float64) - float(md)).sum())
        for g in range(zt.size // 32):
            zg, dg = zt[32 * g: 32 * g + 32], zd[32 * g: 32 * g + 32]
            pm = _p(np.array([zg.max()], F32), ml, inv_s, -EX2_ERR)[0]
            rb = F32(F32(pm * SCALE) + FLOOR)
            p = _p(zg, ml, inv_s, +EX2_ERR)
            r = np.maximum((p + _p(dg, mld, ninv_sd, 0.0)).astype(F32), F32(0))
            acc = _group_sum(r)
            if acc <= 0:
                continue
            for word in rng.integers(0, 2 ** 32, 6, dtype=np.uint64):
                u = F32(float(int(word) >> 8) * 2.0 ** -24)
                e = F32(-np.log1p(-np.float64(u)))   # log1p: within an ulp, as CUDA's log1pf
                e = F32(e * F32(1.0 - 2.0 ** -23))    # and rounded down by one ulp at worst
                key = F32(e / acc)
                lb = float(u) / float(rb)
                for k1 in (lb * 0.99, lb * (1 - 2e-5), lb * (1 - 1.1e-5), lb, lb * 1.00001):
                    k1 = F32(k1)
                    if F32(u * FILTER) > F32(k1 * rb):
                        skipped += 1
                        assert key > k1, (g, float(key), float(k1))
    assert skipped > 1000
