"""Seeded input generators: determinism, rounding, shapes and recipe structure."""
import numpy as np
import pytest
import torch

from paper_2508_15371_gb300 import workloads as W


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.normal(0, 10, 100000).astype(np.float32),
                        np.array([0.0, -0.0, np.inf, -np.inf, 1e-40, 3.0e38], np.float32)])
    ours = W.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    back = W.bf16_bits_to_f32(ours)
    assert np.array_equal(back, torch.from_numpy(x).to(torch.bfloat16).float().numpy())


@pytest.mark.parametrize("name,kw", [("c1", dict(B=1, K=4, V=1000)), ("c2", dict(B=3, K=8, V=640)),
                                     ("c3", dict(B=2, K=8, V=2048)), ("c4", dict(B=2, K=16, V=1536))])
def test_recipes_deterministic_and_shaped(name, kw):
    a = W.make(name, **kw)
    b = W.make(name, threads=1, **kw)
    assert a.draft.shape == (kw["B"], kw["K"], kw["V"]) == a.target.shape
    assert a.tokens.shape == (kw["B"], kw["K"]) and a.tokens.dtype == np.int32
    assert np.array_equal(a.draft, b.draft) and np.array_equal(a.target, b.target)
    assert np.array_equal(a.tokens, b.tokens)
    assert a.tokens.min() >= 0 and a.tokens.max() < kw["V"]
    assert a.draft.dtype == (np.float32 if a.dtype == "f32" else np.uint16)


def test_c1_drafted_tokens_are_argmax():
    w = W.make("c1", V=5000)
    assert np.array_equal(w.tokens, np.argmax(w.draft, axis=-1))


def test_c3_profile_readings():
    r = W.zipf_profile(10, "rank")
    assert r[0] == np.float32(4.0) and np.all(np.diff(r) < 0)
    l = W.zipf_profile(10, "log")
    assert l[0] == 0.0 and l[1] == pytest.approx(-4.4 * np.log(2), rel=1e-6)


def test_c5_generator_tables():
    t = W.normal_table()
    assert t.shape == (1 << W.NORMAL_BITS,) == (8192,) and t.dtype == np.float32
    assert np.all(np.diff(t) > 0) and abs(float(t.mean())) < 1e-6
    assert float(t.std()) == pytest.approx(1.0, abs=2e-3)
    h = W.ar1_heights(32, 200, seed=4, table=t)
    assert h.shape == (200, 32) and h.min() >= 0 and h.max() <= 12
    assert abs(float(h.mean()) - 6.0) < 1.0
    d, tg, tok = W.decode_row_host(t, h, 3, 5, 2, 16, 32000)
    assert d.dtype == np.float32 and tok == int(np.argmax(d))
    d2, _, _ = W.decode_row_host(t, h, 3, 5, 2, 16, 32000)
    assert np.array_equal(d, d2)
    d3, _, _ = W.decode_row_host(t, h, 4, 5, 2, 16, 32000)
    assert not np.array_equal(d, d3)
