"""Pins of the LM-head oracle (oracle/lmhead.py) against values fixed by the
mathematics: a hand-worked product, the triple-loop definition of z = h W^T,
one-hot weights that select hidden coordinates, the uniform and spike closed
forms of Sec. III.B(1) reached through the head, and the first-order error
bound of the signals."""
import math

import numpy as np
import pytest

import oracle as O
from paper_2508_15371_gb300 import workloads as W


def bits(x):
    return W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def test_hand_worked_product():
    # h = [[1, 2], [0, -1]], W = [[1, 0], [1, 1], [0, 3]]  ->  z = [[1, 3, 6], [0, -1, -3]]
    z = O.lm_head_logits(bits([[1, 2], [0, -1]]), bits([[1, 0], [1, 1], [0, 3]]))
    assert np.array_equal(z, [[1.0, 3.0, 6.0], [0.0, -1.0, -3.0]])


def test_triple_loop_definition():
    rng = np.random.default_rng(3)
    h = rng.integers(-8, 9, size=(3, 5)) / 8.0
    w = rng.integers(-8, 9, size=(7, 5)) / 4.0
    z = O.lm_head_logits(bits(h), bits(w))
    for r in range(3):
        for v in range(7):
            acc = 0.0
            for j in range(5):
                acc += float(h[r, j]) * float(w[v, j])
            assert z[r, v] == acc


def test_one_hot_weights_select_hidden_coordinates():
    d, V = 16, 40
    rng = np.random.default_rng(4)
    h = rng.integers(-64, 65, size=(4, d)) / 32.0
    w = np.zeros((V, d))
    col = np.arange(V) % d
    c = rng.integers(1, 4, size=V).astype(float)
    w[np.arange(V), col] = c
    z = O.lm_head_logits(bits(h), bits(w))
    assert np.array_equal(z, h[:, col] * c)


def test_zero_hidden_gives_uniform_row():
    V = 1000
    out = O.lm_head_confidence(bits(np.zeros((2, 8))), bits(np.ones((V, 8))), O.Params())
    assert np.allclose(out["H"], math.log(V), rtol=0, atol=1e-12)
    assert np.all(out["margin"] == 0) and np.all(out["psm"] == 0) and np.all(out["argmax"] == 0)
    assert np.all(out["argmax_flag"])       # a tie: the argmax is flagged


@pytest.mark.parametrize("a", [0.5, 4.0, 8.0])
def test_spike_through_the_head(a):
    # h = a e_0 and one weight row e_0: logit a at v*, 0 elsewhere
    V, d, vs = 512, 4, 137
    h = np.zeros((1, d)); h[0, 0] = a
    w = np.zeros((V, d)); w[vs, 0] = 1.0
    out = O.lm_head_confidence(bits(h), bits(w), O.Params())
    S = math.exp(a) + V - 1
    H = math.log(S) - a * math.exp(a) / S
    assert out["argmax"][0] == vs and out["margin"][0] == a
    assert out["H"][0] == pytest.approx(H, abs=1e-12)
    assert out["lse"][0] == pytest.approx(math.log(S), abs=1e-12)
    assert out["psm"][0] == pytest.approx((math.exp(a) - 1) / S, abs=1e-12)


def test_signal_error_bound_holds():
    rng = np.random.default_rng(5)
    V, eps = 300, 1e-4
    P = O.Params(beta_sig=2.0)
    for _ in range(40):
        z = rng.standard_normal(V) * rng.uniform(0.1, 4)
        z[rng.integers(V)] += rng.uniform(0, 10)
        s0 = O.drafter_signals(z)
        s1 = O.drafter_signals(z + rng.uniform(-eps, eps, V))
        c0 = O.unified_confidence(s0["H"], s0["margin"], s0["psm"], V, P)
        c1 = O.unified_confidence(s1["H"], s1["margin"], s1["psm"], V, P)
        b = O.signal_error_bound(eps, s0["H"], V, P.lam, P.beta_sig)
        slack = 1.01       # second-order terms
        assert abs(s1["lse"] - s0["lse"]) <= b["lse"] * slack
        assert abs(s1["H"] - s0["H"]) <= b["H"] * slack
        assert abs(s1["psm"] - s0["psm"]) <= b["psm"] * slack
        assert abs(c1 - c0) <= b["conf"] * slack
        if s0["argmax"] == s1["argmax"]:
            assert abs(s1["margin"] - s0["margin"]) <= b["margin"] * slack


def test_exact_recipe_is_exact_in_float32():
    # the exact recipe's dot products have every partial sum representable in
    # float32, so a float32 accumulation in any order gives the float64 value
    w = W.make_lmhead(R=5, d=256, V=300, seed=1, exact=True)
    z = O.lm_head_logits(w.hidden, w.weight)
    h32 = W.bf16_bits_to_f32(w.hidden)
    w32 = W.bf16_bits_to_f32(w.weight)
    rng = np.random.default_rng(0)
    for r in range(5):
        for v in rng.integers(0, 300, size=20):
            order = rng.permutation(256)
            acc = np.float32(0)
            for j in order:
                acc = np.float32(acc + np.float32(h32[r, j] * w32[v, j]))
            assert float(acc) == z[r, v]


def test_spiked_rows_peak_at_their_token():
    w = W.make_lmhead(R=16, d=256, V=2000, seed=2)
    out = O.lm_head_confidence(w.hidden, w.weight, O.Params())
    z = out["logits"]
    for r in range(16):
        v = w.spike_token[r]
        if v >= 0:
            # the spike raises z[r, v] by its height over the row's noise level
            assert z[r, v] > np.median(z[r])
