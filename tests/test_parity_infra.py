"""The parity machinery itself, on the CPU: the pooled oracle gives the same
result as the oracle called directly (same Philox counters for every
sequence), `compare` catches planted mistakes, and the flag bound rejects an
oracle that flags everything."""
import numpy as np
import pytest

import oracle as O
import oracle_pool
from parity_util import assert_flag_bound, compare, decisions_total
from paper_2508_15371_gb300 import workloads as W


def _pdict(rule):
    return dict(k_min=1, k_max=6, lam=(1 / 3, 1 / 3, 1 / 3), beta_sig=1.0,
                beta_rank=3 if rule == "paper" else 0, alpha=1.0, tau_base=0.1, gamma=1.0,
                tau_sign=1, rule=rule)


def _as_gpu_dict(r):
    """An oracle result shaped like the library's outputs."""
    return {"H": r.H.astype(np.float32), "margin": r.margin.astype(np.float32),
            "conf": r.conf.astype(np.float32), "lse": r.lse.astype(np.float32),
            "argmax": r.argmax, "k_next": r.k_next, "n_accept": r.n_accept,
            "out_tokens": r.out_tokens, "accept": r.accept.astype(np.uint8)}


@pytest.fixture(scope="module")
def small():
    return W.make("c2", B=7, K=6, V=700)


@pytest.mark.parametrize("rule", ["paper", "sampled"])
def test_pool_matches_direct_oracle(small, rule):
    w = small
    k_row = np.array([6, 0, 3, 6, 1, 5, 2])
    d = O.logits_to_f64(w.draft, w.dtype)
    t = O.logits_to_f64(w.target, w.dtype)
    direct = O.confidence_verify(d, t, w.tokens, O.Params(**_pdict(rule)), seed=9, iteration=5, k_row=k_row)
    pooled = oracle_pool.fused(w, _pdict(rule), 9, iteration=5, k_row=k_row, chunk=2)
    for name in ("H", "margin", "conf", "lse"):
        assert np.array_equal(np.nan_to_num(getattr(direct, name), nan=-7.0),
                              np.nan_to_num(getattr(pooled, name), nan=-7.0)), name
    for name in ("argmax", "k_next", "n_accept", "out_tokens", "accept", "tok_flag", "n_flag"):
        assert np.array_equal(getattr(direct, name), getattr(pooled, name)), name


def test_compare_catches_planted_mistakes(small):
    w = small
    r = oracle_pool.fused(w, _pdict("sampled"), 3, iteration=1)
    g = _as_gpu_dict(r)
    f = compare(w, g, r)
    assert f["seqs"] == w.B and decisions_total(f) == 3 * w.B + w.B * w.K
    assert max(f["max_abs_err"].values()) < 1e-6
    for name, mutate in [
        ("H", lambda g: g["H"].__setitem__((2, 1), g["H"][2, 1] + 3e-4)),
        ("argmax", lambda g: g["argmax"].__setitem__((0, 0), g["argmax"][0, 0] + 1)),
        ("n_accept", lambda g: g["n_accept"].__setitem__(4, (g["n_accept"][4] + 1) % (w.K + 1))),
        ("out_tokens", lambda g: g["out_tokens"].__setitem__((5, 0), -5)),
        ("k_next", lambda g: g["k_next"].__setitem__(1, g["k_next"][1] % 6 + 1)),
    ]:
        bad = {k: v.copy() for k, v in g.items()}
        mutate(bad)
        with pytest.raises(AssertionError):
            compare(w, bad, r)


def test_flag_bound_rejects_an_oracle_that_flags_everything():
    ok = {"k": 1, "n": 0, "tok": 0, "acc": 0, "seqs": 64, "rows": 512}
    assert_flag_bound(ok)
    bad = dict(ok, k=64, n=64, tok=64, acc=512)
    with pytest.raises(AssertionError):
        assert_flag_bound(bad)
