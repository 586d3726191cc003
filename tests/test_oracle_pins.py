"""Pins for the CPU oracle against things other than itself.

Closed forms, the paper's own limit statements (tests/golden/paper_statements.json),
independent library routines (scipy), brute force on tiny inputs, and exact
laws of the sampled rule at V = 8.  Each test is chosen so that a plausible
slip in the oracle (a dropped term, a wrong sign, a transposed operand, an
off-by-one in the prefix scan) fails it.
"""
import json
import math
import os

import numpy as np
import pytest
import scipy.special as sps
import scipy.stats as st

import oracle as O

GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_statements.json")))


def P(**kw):
    base = dict(k_min=1, k_max=8, lam=(1 / 3, 1 / 3, 1 / 3), beta_sig=1.0, beta_rank=3,
                alpha=1.0, tau_base=0.1, gamma=1.0, tau_sign=1, rule="paper")
    base.update(kw)
    return O.Params(**base)


# ---------------------------------------------------------------- entropy etc.

@pytest.mark.parametrize("V", [2, 8, 1000, 32000])
def test_uniform_row_has_max_entropy(V):
    # Sec. III.B(1): log|V| is the entropy of the uniform distribution
    s = O.drafter_signals(np.zeros(V))
    assert s["H"] == pytest.approx(math.log(V), abs=1e-12)
    assert s["margin"] == 0.0
    assert s["psm"] == pytest.approx(0.0, abs=1e-15)
    assert s["argmax"] == 0
    C = O.unified_confidence(s["H"], s["margin"], s["psm"], V, P())
    # entropy term 0, sigmoid(0) = 1/2, softmax margin 0
    assert C == pytest.approx(0.5 / 3, abs=1e-12)


@pytest.mark.parametrize("V,h", [(8, 0.5), (8, 3.0), (1000, 2.0), (32000, 7.5), (32000, 20.0)])
def test_spike_closed_form(V, h):
    z = np.zeros(V)
    z[V // 3] = h
    s = O.drafter_signals(z)
    a = (V - 1) * math.exp(-h)
    H = math.log1p(a) + h * a / (1 + a)
    assert s["H"] == pytest.approx(H, rel=1e-11, abs=1e-13)
    assert s["margin"] == pytest.approx(h, abs=0)
    assert s["psm"] == pytest.approx((1 - math.exp(-h)) / (1 + a), rel=1e-12)
    assert s["argmax"] == V // 3
    assert s["lse"] == pytest.approx(h + math.log1p(a), rel=1e-12)


def test_dominant_spike_limits():
    V = 32000
    z = np.zeros(V)
    z[5] = 60.0
    s = O.drafter_signals(z)
    assert s["H"] < 1e-18          # H -> 0 (about 60 * V * e^-60)
    assert s["margin"] == 60.0     # margin -> spike gap
    assert O.unified_confidence(s["H"], s["margin"], s["psm"], V, P()) == 1.0


def test_two_equal_maxima():
    V = 5000
    z = np.zeros(V)
    z[[7, 4000]] = 40.0
    s = O.drafter_signals(z)
    assert s["H"] == pytest.approx(math.log(2), rel=1e-9)
    assert s["margin"] == 0.0
    assert s["argmax"] == 7        # lowest index (reading C8)
    assert s["psm"] == pytest.approx(0.0, abs=1e-15)


def test_entropy_matches_scipy_on_random_rows():
    rng = np.random.default_rng(11)
    for V in (8, 97, 4096):
        for scale in (0.1, 1.0, 5.0):
            z = rng.normal(0, scale, V)
            s = O.drafter_signals(z)
            p = sps.softmax(z)
            assert s["H"] == pytest.approx(st.entropy(p), rel=1e-12, abs=1e-14)
            assert s["lse"] == pytest.approx(sps.logsumexp(z), rel=1e-13)


def test_masked_logits_carry_no_probability():
    rng = np.random.default_rng(5)
    z = rng.normal(0, 1, 64)
    zm = z.copy()
    zm[10:20] = -np.inf
    s = O.drafter_signals(zm)
    keep = np.r_[z[:10], z[20:]]
    assert s["H"] == pytest.approx(st.entropy(sps.softmax(keep)), rel=1e-12)
    one = np.full(16, -np.inf)
    one[3] = 1.0
    s1 = O.drafter_signals(one)
    assert s1["H"] == 0.0 and s1["margin"] == np.inf and s1["argmax"] == 3


def test_margins_by_sorting():
    rng = np.random.default_rng(7)
    for _ in range(50):
        V = int(rng.integers(2, 12))
        z = rng.integers(-3, 4, V).astype(float)      # many ties
        s = O.drafter_signals(z)
        order = np.argsort(-z, kind="stable")          # stable: lowest index first among ties
        assert s["argmax"] == order[0]
        assert s["margin"] == z[order[0]] - z[order[1]]
        p = sps.softmax(z)
        assert s["psm"] == pytest.approx(p[order[0]] - p[order[1]], abs=1e-15)


def test_unified_confidence_components():
    V = 100
    # each lambda one-hot picks one normalised signal (Table III single-signal ablations)
    H, margin, psm = 2.0, 1.5, 0.3
    c_ent = O.unified_confidence(H, margin, psm, V, P(lam=(1, 0, 0)))
    c_mar = O.unified_confidence(H, margin, psm, V, P(lam=(0, 1, 0)))
    c_soft = O.unified_confidence(H, margin, psm, V, P(lam=(0, 0, 1)))
    assert c_ent == pytest.approx(1 - H / math.log(V))
    assert c_mar == pytest.approx(sps.expit(margin))
    assert c_soft == pytest.approx(psm * V / (V - 1))
    assert O.unified_confidence(H, margin, psm, V, P(lam=(0.2, 0.5, 0.3))) == pytest.approx(
        0.2 * c_ent + 0.5 * c_mar + 0.3 * c_soft)
    # the sigmoid is the logistic function with sharpness beta_sig, range (0, 1)
    lo, hi = GOLD["sigmoid_range"]["low"], GOLD["sigmoid_range"]["high"]
    for m in (0.0, 0.01, 2.0, 30.0):
        c = O.unified_confidence(0.0, m, 0.0, V, P(lam=(0, 1, 0), beta_sig=2.5))
        assert lo < c <= hi and c == pytest.approx(sps.expit(2.5 * m))
    # clamp to [0, 1] (the softmax margin term alone can exceed 1)
    assert O.unified_confidence(0.0, 50.0, 1.0, V, P()) == 1.0


# ---------------------------------------------------------------- draft length

def test_draft_length_paper_limits():
    for kmax in (4, 8, 16):
        for alpha in (1.0, 0.75, 0.5):
            pp = P(k_max=kmax, k_min=1, alpha=alpha)
            k1, _ = O.next_draft_length([1.0] * 5, pp)            # Cbar -> 1
            assert k1 == min(kmax, max(1, math.floor(alpha * kmax)))
            k0, _ = O.next_draft_length([0.0] * 5, pp)            # Cbar -> 0
            assert k0 == 1
    pp = P(k_max=16, k_min=3)
    assert O.next_draft_length([0.0, 0.01], pp)[0] == 3           # clipped at k_min
    assert O.next_draft_length([], pp)[0] == 3


def test_draft_length_monotone_and_bounded():
    pp = P(k_max=16, k_min=2, alpha=0.9)
    grid = np.linspace(0, 1, 2001)
    ks = [O.next_draft_length([c, c], pp)[0] for c in grid]
    assert all(2 <= k <= 16 for k in ks)
    assert all(b >= a for a, b in zip(ks, ks[1:]))
    # mean over the window, not the last or first position
    assert O.next_draft_length([1.0, 0.0, 0.5, 0.5], P(k_max=8))[0] == 4


def test_draft_length_flags_integer_boundaries():
    pp = P(k_max=10)
    k, flag = O.next_draft_length([0.3], pp)      # 0.3 * 10 sits on 3
    assert flag
    k, flag = O.next_draft_length([0.35], pp)
    assert not flag and k == 3


# ---------------------------------------------------------------- PAPER rule

def test_threshold_endpoints():
    pp = P(tau_base=GOLD["tau_base_example"]["value"], gamma=0.7)
    assert O.tau_t(1.0, pp) == pytest.approx(0.1)
    assert O.tau_t(0.0, pp) == pytest.approx(0.8)
    pn = P(tau_base=0.1, gamma=0.7, tau_sign=-1)               # prose reading
    assert O.tau_t(1.0, pn) == pytest.approx(0.8)
    assert O.tau_t(0.0, pn) == pytest.approx(0.1)


def test_beta1_is_exact_match_on_tie_free_rows():
    rng = np.random.default_rng(3)
    for _ in range(200):
        V = 8
        zt = rng.normal(0, 2, V)
        tok = int(rng.integers(0, V))
        acc, _ = O.accept_paper(zt, tok, tau=0.0, beta_rank=1)
        assert acc == (tok == int(np.argmax(zt)))


def test_fixed_tau_rule_by_sorting():
    rng = np.random.default_rng(4)
    for _ in range(300):
        V = 8
        zt = rng.normal(0, 1.5, V)
        tok = int(rng.integers(0, V))
        beta = int(rng.integers(1, 5))
        tau = float(rng.uniform(0, 2))
        acc, _ = O.accept_paper(zt, tok, tau, beta)
        rank = int(np.where(np.argsort(-zt) == tok)[0][0])       # 0 = top-1 (no ties)
        lp = sps.log_softmax(zt)
        want = rank < beta and (lp.max() - lp[tok]) <= tau
        assert acc == want
        # gamma = 0 makes tau independent of the confidence
        pp = P(gamma=0.0, tau_base=tau)
        assert O.tau_t(0.0, pp) == O.tau_t(1.0, pp) == tau


def test_rank_gate_counts_strictly_greater():
    zt = np.array([1.0, 3.0, 3.0, 2.0, 3.0])
    assert O.rank_gate(zt, 2, 1)           # ties with the max are inside the top-1
    assert not O.rank_gate(zt, 3, 3)       # three logits above
    assert O.rank_gate(zt, 3, 4)
    assert O.rank_gate(zt, 0, 0)           # beta = 0: no gate


def _seq(acc_pattern, rule="paper"):
    """A sequence whose per-position PAPER decisions follow acc_pattern exactly."""
    K = len(acc_pattern)
    V = 8
    d = np.zeros((K, V))
    t = np.zeros((K, V))
    toks = np.arange(K) % V
    for i, a in enumerate(acc_pattern):
        t[i, toks[i]] = 5.0 if a else -5.0       # top-1 (accept) or far below (reject)
        t[i, (toks[i] + 1) % V] = 1.0
    return d, t, toks


@pytest.mark.parametrize("pattern", [
    [1, 1, 1, 1], [0, 1, 1, 1], [1, 0, 1, 0], [1, 1, 1, 0], [1], [0]])
def test_halt_at_first_failure(pattern):
    d, t, toks = _seq(pattern)
    K = len(pattern)
    conf = np.full(K, 0.5)
    v = O.verify_sequence(d, t, toks, conf, K, P(k_max=K), 0, 0, 0)
    n = pattern.index(0) if 0 in pattern else K
    assert v["n_accept"] == n
    out = v["out_tokens"]
    assert list(out[:n]) == list(toks[:n])
    if n < K:
        assert out[n] == int(np.argmax(t[n]))      # verifier's greedy token
        assert all(out[n + 1:] == -1)
    else:
        assert len(out) == K                       # no bonus token (reading C10)


def test_ragged_window_only_uses_present_positions():
    d, t, toks = _seq([1, 1, 0, 0])
    conf = np.full(4, 0.5)
    v = O.verify_sequence(d, t, toks, conf, 2, P(k_max=4), 0, 0, 0)
    assert v["n_accept"] == 2 and list(v["out_tokens"]) == [toks[0], toks[1], -1, -1]
    v0 = O.verify_sequence(d, t, toks, conf, 0, P(k_max=4), 0, 0, 0)
    assert v0["n_accept"] == 0 and list(v0["out_tokens"]) == [-1] * 4


# ---------------------------------------------------------------- SAMPLED rule

def _rows8(rng, V=8):
    zt = rng.normal(0, 1.2, V)
    zd = zt + rng.normal(0, 0.9, V)
    return zt, zd


@pytest.mark.parametrize("tau", [0.0, 0.3])
def test_sampled_acceptance_probability(tau):
    # the measure of {u in [0,1): accept} equals min(1, e^tau p / q)
    rng = np.random.default_rng(8)
    zt, zd = _rows8(rng)
    p, q = sps.softmax(zt), sps.softmax(zd)
    us = (np.arange(1 << 14) + 0.5) / (1 << 14)
    for x in range(8):
        frac = np.mean([O.accept_sampled(zt, zd, x, tau, u, 0)[0] for u in us])
        assert frac == pytest.approx(min(1.0, math.exp(tau) * p[x] / q[x]), abs=2.0 / (1 << 14))


def test_residual_race_law():
    rng = np.random.default_rng(9)
    zt, zd = _rows8(rng)
    p, q = sps.softmax(zt), sps.softmax(zd)
    r = np.maximum(0, p - q)
    n = 6000
    counts = np.zeros(8)
    for it in range(n):
        tok, _ = O.residual_token(zt, zd, 123, 0, 0, it)
        counts[tok] += 1
    assert counts[r == 0].sum() == 0
    exp = r / r.sum() * n
    m = exp > 0
    chi2 = ((counts[m] - exp[m]) ** 2 / exp[m]).sum()
    assert st.chi2.sf(chi2, m.sum() - 1) > 1e-3


@pytest.mark.parametrize("tau", [0.0, 0.4])
def test_sampled_output_law_by_enumeration(tau):
    # law(y) = q(y) a(y) + (sum_x q(x)(1 - a(x))) r(y)/sum r, with a and the
    # residual law both measured from the oracle's own decisions; tau = 0 must
    # give the target law p exactly (speculative sampling, reading C9).
    rng = np.random.default_rng(10)
    zt, zd = _rows8(rng)
    p, q = sps.softmax(zt), sps.softmax(zd)
    # acceptance measure from the oracle's decision rule (exact: piecewise in u)
    a = np.array([min(1.0, math.exp(tau) * p[x] / q[x]) for x in range(8)])
    for x in range(8):
        u_edge = a[x]
        if u_edge < 1:
            assert O.accept_sampled(zt, zd, x, tau, u_edge * 0.999999, 0)[0]
            assert not O.accept_sampled(zt, zd, x, tau, min(u_edge * 1.000001, 0.9999999), 0)[0]
    r = np.maximum(0, p - q)
    law = q * a + (q * (1 - a)).sum() * r / r.sum()
    assert law.sum() == pytest.approx(1.0, abs=1e-15)
    if tau == 0.0:
        assert np.max(np.abs(law - p)) < 1e-15
    else:
        closed = np.minimum(q, math.exp(tau) * p) + (1 - np.minimum(q, math.exp(tau) * p).sum()) * r / r.sum()
        assert np.max(np.abs(law - closed)) < 1e-15


def test_sampled_pipeline_reproduces_target_law():
    # Monte Carlo through verify_sequence: draft x ~ q, K = 1, tau = 0 -> output ~ p
    rng = np.random.default_rng(12)
    V = 8
    zt, zd = _rows8(rng, V)
    p, q = sps.softmax(zt), sps.softmax(zd)
    pp = P(k_max=1, rule="sampled", beta_rank=0, tau_base=0.0, gamma=0.0)
    n = 6000
    xs = rng.choice(V, size=n, p=q)
    counts = np.zeros(V)
    for it in range(n):
        v = O.verify_sequence(zd[None], zt[None], np.array([xs[it]]), np.array([0.5]), 1, pp, 77, 0, it)
        counts[v["out_tokens"][0]] += 1
    chi2 = ((counts - p * n) ** 2 / (p * n)).sum()
    assert st.chi2.sf(chi2, V - 1) > 1e-3


def test_sampled_flags_near_threshold():
    zt = np.log(np.array([0.5, 0.25, 0.25]))
    zd = np.log(np.array([0.25, 0.5, 0.25]))
    # u * q == e^tau * p at u = 0.5 for token 1 with tau = 0
    acc, flag, p, q = O.accept_sampled(zt, zd, 1, 0.0, 0.5, 0)
    assert flag and not acc
    acc, flag, _, _ = O.accept_sampled(zt, zd, 1, 0.0, 0.4, 0)
    assert acc and not flag


def test_residual_race_law_across_groups():
    # V = 100 spans four groups of 32 (the last one partial): the two-level
    # race must still give each entry probability r_v / sum(r)
    rng = np.random.default_rng(19)
    V = 100
    zt = rng.normal(0, 1.0, V)
    zd = zt + rng.normal(0, 1.0, V)
    p, q = sps.softmax(zt), sps.softmax(zd)
    r = np.maximum(0, p - q)
    n = 20000
    counts = np.zeros(V)
    for it in range(n):
        tok, _ = O.residual_token(zt, zd, 7, 1, 2, it)
        counts[tok] += 1
    assert counts[r == 0].sum() == 0
    # compare group masses (enough counts per cell) and the within-group law
    G = O.philox.GROUP
    gm = np.array([r[i:i + G].sum() for i in range(0, V, G)]) / r.sum() * n
    gc = np.array([counts[i:i + G].sum() for i in range(0, V, G)])
    chi2 = ((gc - gm) ** 2 / gm).sum()
    assert st.chi2.sf(chi2, len(gm) - 1) > 1e-3
    top = np.argsort(-r)[:8]
    e = r[top] / r.sum() * n
    chi2 = ((counts[top] - e) ** 2 / e).sum()
    assert st.chi2.sf(chi2, len(top)) > 1e-4


def test_residual_falls_back_to_target_argmax_when_empty():
    z = np.array([0.1, 2.0, -1.0, 0.5])
    tok, flag = O.residual_token(z, z, 0, 0, 0, 0)
    assert tok == 1 and not flag


# ---------------------------------------------------------------- whole iteration

def test_confidence_verify_consistency_small_batch():
    from paper_2508_15371_gb300 import workloads as W
    w = W.make("c2", B=3, K=4, V=257)
    d = O.logits_to_f64(w.draft, w.dtype)
    t = O.logits_to_f64(w.target, w.dtype)
    for rule, beta in (("paper", 3), ("sampled", 0)):
        pp = P(k_max=4, rule=rule, beta_rank=beta)
        r = O.confidence_verify(d, t, w.tokens, pp, seed=1, iteration=2)
        for b in range(3):
            n = r.n_accept[b]
            assert 0 <= n <= 4
            assert all(r.accept[b, :n]) and (n == 4 or not r.accept[b, n])
            assert list(r.out_tokens[b, :n]) == list(w.tokens[b, :n])
            k, _ = O.next_draft_length(r.conf[b], pp)
            assert r.k_next[b] == k


def test_decode_sim_replay_feeds_k_forward():
    from paper_2508_15371_gb300 import workloads as W
    table = W.normal_table()
    heights = W.ar1_heights(2, 6, seed=4, table=table)

    def gen(it, b, k):
        return W.decode_iteration_host(table, heights, it, b, k, 16, 512, seed=4)

    pp = P(k_max=16, k_min=1, rule="sampled", beta_rank=0)
    traj = O.decode_sim_sequence(gen, 1, 6, 16, pp, 4)
    assert traj[0]["k"] == 16
    for a, b in zip(traj, traj[1:]):
        assert b["k"] == a["k_next"]
    for s in traj:
        assert 1 <= s["k_next"] <= 16 and 0 <= s["n_accept"] <= s["k"]


# ---------------------------------------------------------------- fixed k, bonus row

def test_fixed_draft_length_ignores_confidence():
    # Table III, "fixed k": the draft length no longer follows the confidence
    pp = P(k_max=16, k_min=2, k_fixed=9)
    for window in ([0.0] * 4, [1.0] * 4, [0.3, 0.9], []):
        assert O.next_draft_length(window, pp) == (9, False)


def test_bonus_argmax_by_sorting():
    rng = np.random.default_rng(30)
    for _ in range(20):
        z = np.round(rng.normal(0, 1, 50), 1)          # ties are common at one decimal
        tok, flag = O.bonus_token(z, "paper", 0, 0, 0, 0)
        top = max(z)
        assert tok == min(i for i in range(50) if z[i] == top) and not flag


@pytest.mark.parametrize("V", [8, 100])
def test_bonus_draw_has_the_verifier_law(V):
    # the sampled bonus token is the two-level race with r = p: its law is p
    # (V = 100 spans four groups of 32, the last one partial)
    rng = np.random.default_rng(31 + V)
    zt = rng.normal(0, 1.0, V)
    p = sps.softmax(zt)
    n = 20000
    counts = np.zeros(V)
    for it in range(n):
        tok, _ = O.bonus_token(zt, "sampled", 5, 3, 4, it)
        counts[tok] += 1
    if V == 8:
        chi2 = ((counts - p * n) ** 2 / (p * n)).sum()
        assert st.chi2.sf(chi2, V - 1) > 1e-3
    else:
        G = O.philox.GROUP
        gm = np.array([p[i:i + G].sum() for i in range(0, V, G)]) * n
        gc = np.array([counts[i:i + G].sum() for i in range(0, V, G)])
        assert st.chi2.sf(((gc - gm) ** 2 / gm).sum(), len(gm) - 1) > 1e-3
        top = np.argsort(-p)[:8]
        e = p[top] * n
        assert st.chi2.sf(((counts[top] - e) ** 2 / e).sum(), len(top)) > 1e-4


def test_bonus_row_follows_an_accepted_window():
    # K = 1, tau = 0, the verifier's extra row present: when the draft is
    # accepted the second emitted token follows the extra row's law p1; when
    # it is rejected only the correction is emitted (no bonus)
    rng = np.random.default_rng(33)
    V = 8
    zt, zd = _rows8(rng, V)
    z1 = rng.normal(0, 1.0, V)
    p1 = sps.softmax(z1)
    pp = P(k_max=1, rule="sampled", beta_rank=0, tau_base=0.0, gamma=0.0, bonus=True)
    n = 6000
    xs = rng.choice(V, size=n, p=sps.softmax(zd))
    counts = np.zeros(V)
    for it in range(n):
        v = O.verify_sequence(zd[None], np.stack([zt, z1]), np.array([xs[it]]), np.array([0.5]), 1, pp, 78, 0, it)
        out = v["out_tokens"]
        assert out.shape == (2,)
        if v["n_accept"] == 1:
            assert out[0] == xs[it] and 0 <= out[1] < V
            counts[out[1]] += 1
        else:
            assert out[1] == -1
    m = counts.sum()
    assert m > 1000
    chi2 = ((counts - p1 * m) ** 2 / (p1 * m)).sum()
    assert st.chi2.sf(chi2, V - 1) > 1e-3
    # PAPER rule: the bonus token is the extra row's argmax
    pq = P(k_max=1, rule="paper", beta_rank=0, tau_base=100.0, gamma=0.0, bonus=True)
    v = O.verify_sequence(zd[None], np.stack([zt, z1]), np.array([0]), np.array([0.5]), 1, pq, 0, 0, 0)
    assert v["n_accept"] == 1 and v["out_tokens"][1] == int(np.argmax(z1))
