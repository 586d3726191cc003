"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Sizes span many warps' slices, row boundaries inside slices and ragged row
tails; the full-size cases run the launch configuration bench.py times and
check sampled sequences against the oracle plus size-independent properties
everywhere else.
"""
import numpy as np
import pytest

from parity_util import check_properties, compare, gpu_fused, oracle_fused

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def cmsd():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2508_15371_gb300 import cmsd as c
    c.lib()
    return c


@pytest.fixture(scope="module")
def W():
    from paper_2508_15371_gb300 import workloads
    return workloads


RULES = [("paper", dict(beta_rank=3)), ("sampled", dict(beta_rank=0))]


@pytest.mark.parametrize("rule,kw", RULES)
@pytest.mark.parametrize("name,size", [
    ("c1", {}),                                   # full size: B1 K4 V32000 f32
    ("c2", {}),                                   # full size: B8 K8 V32128 bf16
    ("c3", dict(B=4)),                            # V = 128256, 32 rows
    ("c4", dict(B=3)),                            # V = 152064, 48 rows
])
def test_parity_configs(cmsd, W, name, size, rule, kw):
    w = W.make(name, **size)
    p = cmsd.params(w.K, rule, **kw)
    g = gpu_fused(cmsd, torch, w, p, iteration=3)
    r = oracle_fused(w, p, iteration=3)
    f = compare(w, g, r)
    print(name, rule, f)


@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_c3_log_profile(cmsd, W, rule, kw):
    w = W.make("c3", B=3, profile="log")
    p = cmsd.params(w.K, rule, **kw)
    compare(w, gpu_fused(cmsd, torch, w, p), oracle_fused(w, p))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [2, 8, 9, 1000, 4099, 32001])
def test_parity_vocab_edges(cmsd, W, V, dtype):
    # odd V: rows start off 16-byte boundaries (head/tail elements)
    w = W.make("c2", B=3, K=5, V=V, dtype=dtype)
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, **kw)
        compare(w, gpu_fused(cmsd, torch, w, p, iteration=7), oracle_fused(w, p, iteration=7))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_parity_ragged_windows(cmsd, W, dtype):
    w = W.make("c2", B=9, K=6, V=3000, dtype=dtype)
    k_row = np.array([6, 0, 1, 3, 6, 2, 0, 5, 4], np.int32)
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, k_min=2, **kw)
        g = gpu_fused(cmsd, torch, w, p, k_row=k_row)
        r = oracle_fused(w, p, k_row=k_row)
        compare(w, g, r, k_row=k_row)
        for b in np.where(k_row == 0)[0]:
            assert g["n_accept"][b] == 0 and np.all(g["out_tokens"][b] == -1)
            assert g["k_next"][b] == 2


@pytest.mark.parametrize("K", [1, 31, 33, 70])
def test_parity_window_lengths(cmsd, W, K):
    w = W.make("c2", B=2, K=K, V=700)
    for rule, kw in RULES:
        p = cmsd.params(K, rule, **kw)
        compare(w, gpu_fused(cmsd, torch, w, p), oracle_fused(w, p))


def test_parity_masked_and_tied_logits(cmsd, W):
    rng = np.random.default_rng(4)
    B, K, V = 2, 4, 1029
    d = rng.normal(0, 1, (B, K, V)).astype(np.float32)
    t = d + rng.normal(0, 0.5, (B, K, V)).astype(np.float32)
    d[0, 0, 100:400] = -np.inf                     # masked vocabulary
    t[0, 0, 100:400] = -np.inf
    d[0, 1, :] = 0.0                               # uniform row: H = log V
    d[0, 2, [5, 900]] = 9.0                        # duplicated maximum: margin 0, argmax 5
    d[1, 0, :] = -np.inf                           # a single finite logit
    d[1, 0, 77] = 1.5
    t[1, 1, [3, 800]] = 20.0                       # tied target maximum
    tok = np.argmax(d, axis=-1).astype(np.int32)
    tok[1, 1] = 800
    from paper_2508_15371_gb300.workloads import Workload, f32_to_bf16_bits
    for dtype in ("f32", "bf16"):
        if dtype == "bf16":
            w = Workload("edge", B, K, V, dtype, f32_to_bf16_bits(d), f32_to_bf16_bits(t), tok, 5)
        else:
            w = Workload("edge", B, K, V, dtype, d, t, tok, 5)
        for rule, kw in RULES:
            p = cmsd.params(K, rule, **kw)
            g = gpu_fused(cmsd, torch, w, p)
            r = oracle_fused(w, p)
            compare(w, g, r)
            assert g["argmax"][0, 2] == 5 and g["margin"][0, 2] == 0.0
            assert np.isinf(g["margin"][1, 0]) and g["argmax"][1, 0] == 77
            assert abs(g["H"][0, 1] - np.log(V)) < 2e-4


def test_exact_match_special_case(cmsd, W):
    # beta = 1, tau = 0: accept iff the drafted token is the verifier argmax
    w = W.make("c2", B=8, K=8, V=2000)
    p = cmsd.params(w.K, "paper", beta_rank=1, tau_base=0.0, gamma=0.0)
    g = gpu_fused(cmsd, torch, w, p)
    tv = (w.target.astype(np.uint32) << 16).view(np.float32)
    for b in range(w.B):
        ztok = np.take_along_axis(tv[b], w.tokens[b][:, None].astype(np.int64), axis=1)[:, 0]
        match = ztok == tv[b].max(axis=-1)          # the draft is a verifier maximum
        n = int(np.argmin(match)) if not match.all() else w.K
        assert g["n_accept"][b] == n


@pytest.mark.parametrize("tau_sign", [1, -1])
def test_parity_tau_readings(cmsd, W, tau_sign):
    w = W.make("c2", B=8, K=8, V=5000)
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, tau_sign=tau_sign, gamma=2.0, **kw)
        compare(w, gpu_fused(cmsd, torch, w, p), oracle_fused(w, p))


def test_separate_entry_points_match_oracle(cmsd, W):
    w = W.make("c3", B=2, V=20000)
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    tok = torch.from_numpy(w.tokens).cuda()
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, **kw)
        c = cmsd.confidence(d, p=p)
        v = cmsd.verify(d, t, tok, c["conf"], draft_lse=c["lse"], p=p, seed=w.seed, iteration=2)
        torch.cuda.synchronize()
        g = {k: x.cpu().numpy() for k, x in {**c, **v}.items()}
        r = oracle_fused(w, p, iteration=2)
        compare(w, g, r)


def test_repeated_calls_reuse_workspace(cmsd, W):
    # counters return to zero after every call: many calls, alternating inputs
    ws_inputs = [W.make("c2", B=4, K=8, V=6000, seed=s) for s in (11, 12)]
    for it in range(6):
        w = ws_inputs[it % 2]
        rule, kw = RULES[it % 2]
        p = cmsd.params(w.K, rule, **kw)
        compare(w, gpu_fused(cmsd, torch, w, p, iteration=it), oracle_fused(w, p, iteration=it))


def test_deterministic(cmsd, W):
    w = W.make("c3", B=4, V=30000)
    p = cmsd.params(w.K, "sampled")
    a = gpu_fused(cmsd, torch, w, p)
    b = gpu_fused(cmsd, torch, w, p)
    for k in a:
        assert np.array_equal(a[k], b[k]), k


def test_device_philox_matches_oracle(cmsd):
    from oracle import philox
    n = 1 << 20
    got = cmsd.philox_fill(0xABCDEF0123, 7, 3, 5, 11, n).cpu().numpy().view(np.uint32)
    c0 = 7 + np.arange(n // 4, dtype=np.uint64)
    want = np.stack(philox.philox4x32_10_np(c0, 3, 5, 11, *philox.seed_key(0xABCDEF0123)), axis=1).reshape(-1)
    assert np.array_equal(got, want)


def test_sampled_rule_reproduces_target_law_on_gpu(cmsd):
    # V = 8, K = 1, tau = 0, no rank gate: emitted token ~ p (speculative sampling)
    from scipy import stats
    rng = np.random.default_rng(21)
    V, B = 8, 4096
    zt = rng.normal(0, 1.2, V).astype(np.float32)
    zd = (zt + rng.normal(0, 0.9, V)).astype(np.float32)
    p = np.exp(zt.astype(np.float64)); p /= p.sum()
    q = np.exp(zd.astype(np.float64)); q /= q.sum()
    d = torch.from_numpy(np.tile(zd, (B, 1, 1))).cuda()
    t = torch.from_numpy(np.tile(zt, (B, 1, 1))).cuda()
    pp = cmsd.params(1, "sampled", tau_base=0.0, gamma=0.0, beta_rank=0)
    counts = np.zeros(V)
    for it in range(12):
        x = rng.choice(V, size=(B, 1), p=q).astype(np.int32)
        o = cmsd.confidence_verify(d, t, torch.from_numpy(x).cuda(), p=pp, seed=99, iteration=it)
        counts += np.bincount(o["out_tokens"][:, 0].cpu().numpy(), minlength=V)
    n = counts.sum()
    chi2 = ((counts - p * n) ** 2 / (p * n)).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-3, (counts / n, p)


# ---------------------------------------------------------------- full sizes

@pytest.mark.parametrize("rule,kw", RULES)
def test_full_size_c3(cmsd, W, rule, kw):
    w = W.make("c3")
    p = cmsd.params(w.K, rule, **kw)
    g = gpu_fused(cmsd, torch, w, p, iteration=1)
    check_properties(w, g, p)
    seqs = [0, 17, 40, 63]
    r = oracle_fused(w, p, iteration=1, seqs=seqs)
    compare(w, g, r, seqs=seqs)


def test_full_size_c4(cmsd, W):
    w = W.make("c4")
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, **kw)
        g = gpu_fused(cmsd, torch, w, p, iteration=1)
        check_properties(w, g, p)
        seqs = [0, 255] if rule == "paper" else [128]
        r = oracle_fused(w, p, iteration=1, seqs=seqs)
        compare(w, g, r, seqs=seqs)
