"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle.

Sizes span many warps' slices, row boundaries inside slices and ragged row
tails; the full-size cases run the launch configuration bench.py times and
check sampled sequences against the oracle plus size-independent properties
everywhere else.
"""
import numpy as np
import pytest

from parity_util import (assert_flag_bound, bonus_view, check_properties, compare, gpu_fused, oracle_fused,
                         record)

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


def test_sampled_rule_modulated_law_on_gpu(cmsd):
    # V = 8, K = 1, tau = 0.4 fixed (gamma = 0), no rank gate: the emitted token
    # has the law of reading C9, min(q, e^tau p) + (1 - sum min(q, e^tau p)) *
    # norm(max(0, p - q)), which differs from p (the drafts are over-accepted)
    from scipy import stats
    rng = np.random.default_rng(33)
    V, B, tau = 8, 4096, 0.4
    zt = rng.normal(0, 1.2, V).astype(np.float32)
    zd = (zt + rng.normal(0, 0.9, V)).astype(np.float32)
    p = np.exp(zt.astype(np.float64)); p /= p.sum()
    q = np.exp(zd.astype(np.float64)); q /= q.sum()
    a = np.minimum(q, np.exp(tau) * p)
    r = np.maximum(0.0, p - q)
    law = a + (1.0 - a.sum()) * r / r.sum()
    assert np.abs(law - p).max() > 0.01                 # the modulation is visible
    d = torch.from_numpy(np.tile(zd, (B, 1, 1))).cuda()
    t = torch.from_numpy(np.tile(zt, (B, 1, 1))).cuda()
    pp = cmsd.params(1, "sampled", tau_base=tau, gamma=0.0, beta_rank=0)
    counts = np.zeros(V)
    for it in range(16):
        x = rng.choice(V, size=(B, 1), p=q).astype(np.int32)
        o = cmsd.confidence_verify(d, t, torch.from_numpy(x).cuda(), p=pp, seed=7, iteration=it)
        counts += np.bincount(o["out_tokens"][:, 0].cpu().numpy(), minlength=V)
    n = counts.sum()
    chi2 = ((counts - law * n) ** 2 / (law * n)).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-3, (counts / n, law)
    chi2_p = ((counts - p * n) ** 2 / (p * n)).sum()
    assert stats.chi2.sf(chi2_p, V - 1) < 1e-6          # and is not the unmodulated law


# ------------------------------------------------ bonus row, fixed draft length

@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_bonus_row(cmsd, W, dtype, rule, kw):
    # the verifier's extra row gives one more token when every draft is
    # accepted; a lenient tau makes that frequent, ragged windows move it
    w = bonus_view(W.make("c2", B=9, K=7, V=2048, dtype=dtype))
    k_row = np.array([6, 0, 1, 3, 6, 2, 6, 5, 4], np.int32)
    bonus_seen = 0
    for extra in (dict(), dict(tau_base=8.0, beta_rank=0)):
        p = cmsd.params(w.K, rule, bonus=1, **{**kw, **extra})
        for kr in (None, k_row):
            g = gpu_fused(cmsd, torch, w, p, iteration=5, k_row=kr)
            r = oracle_fused(w, p, iteration=5, k_row=kr)
            assert g["out_tokens"].shape == (w.B, w.K + 1)
            compare(w, g, r, k_row=kr)
            kb = np.full(w.B, w.K) if kr is None else kr
            bonus_seen += int(sum(g["n_accept"][b] == kb[b] and g["out_tokens"][b, kb[b]] >= 0
                                  for b in range(w.B)))
    assert bonus_seen >= 4


def test_bonus_row_law_on_gpu(cmsd):
    # every draft accepted (tau large): the bonus token of the sampled rule is
    # a draw from the extra verifier row's softmax
    from scipy import stats
    rng = np.random.default_rng(41)
    V, B = 8, 4096
    zt = rng.normal(0, 1.0, V).astype(np.float32)
    z1 = rng.normal(0, 1.3, V).astype(np.float32)
    p1 = np.exp(z1.astype(np.float64)); p1 /= p1.sum()
    d = torch.from_numpy(np.tile(zt, (B, 1, 1))).cuda()
    t = torch.from_numpy(np.tile(np.stack([zt, z1]), (B, 1, 1))).cuda()
    tok = torch.zeros((B, 1), dtype=torch.int32, device="cuda")
    pp = cmsd.params(1, "sampled", tau_base=50.0, gamma=0.0, beta_rank=0, bonus=1)
    counts = np.zeros(V)
    for it in range(8):
        o = cmsd.confidence_verify(d, t, tok, p=pp, seed=11, iteration=it)
        n = o["n_accept"].cpu().numpy()
        assert np.all(n == 1)
        counts += np.bincount(o["out_tokens"][:, 1].cpu().numpy(), minlength=V)
    m = counts.sum()
    chi2 = ((counts - p1 * m) ** 2 / (p1 * m)).sum()
    assert stats.chi2.sf(chi2, V - 1) > 1e-3


@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_fixed_draft_length(cmsd, W, rule, kw):
    w = W.make("c2", B=6, K=8, V=3000)
    for preset in ("fixed_k", "fixed_k_tau"):
        p = cmsd.params(w.K, rule, preset=preset, **kw)
        assert p.k_fixed == w.K
        g = gpu_fused(cmsd, torch, w, p, iteration=2)
        assert np.all(g["k_next"] == w.K)
        compare(w, g, oracle_fused(w, p, iteration=2))
    p = cmsd.params(w.K, rule, k_fixed=3, k_min=2, **kw)
    g = gpu_fused(cmsd, torch, w, p, iteration=2)
    assert np.all(g["k_next"] == 3)
    compare(w, g, oracle_fused(w, p, iteration=2))


@pytest.mark.parametrize("preset", ["entropy_only", "margin_only", "softmax_only", "fixed_tau"])
def test_parity_ablation_presets(cmsd, W, preset):
    w = W.make("c3", B=2, V=20000)
    for rule, kw in RULES:
        p = cmsd.params(w.K, rule, preset=preset, **kw)
        compare(w, gpu_fused(cmsd, torch, w, p, iteration=3), oracle_fused(w, p, iteration=3))


# ------------------------------------------- device error word and guard bands

SENTINEL = {torch.float32: float("nan"), torch.int32: 0x5A5A5A5A, torch.uint8: 0xA5}
GUARD = 64


def _guarded(shape, dtype):
    """A tensor of `shape` inside a larger buffer whose GUARD elements before
    and after hold a sentinel; returns (view, buffer)."""
    n = int(np.prod(shape))
    buf = torch.empty(n + 2 * GUARD, dtype=dtype, device="cuda")
    buf.fill_(SENTINEL[dtype])
    return buf[GUARD:GUARD + n].view(shape), buf


def _guards_intact(buf, dtype):
    h = buf.cpu()
    head, tail = h[:GUARD], h[-GUARD:]
    if dtype == torch.float32:
        return bool(torch.isnan(head).all() and torch.isnan(tail).all())
    return bool((head == SENTINEL[dtype]).all() and (tail == SENTINEL[dtype]).all())


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("rule,kw", RULES)
def test_outputs_stay_inside_their_arrays(cmsd, W, dtype, rule, kw):
    # odd shapes; every output sits between guard bands that must be untouched,
    # and so must the bytes after the workspace
    w = W.make("c2", B=5, K=7, V=1001, dtype=dtype)
    B, K = w.B, w.K
    shapes = {"H": ((B, K), torch.float32), "margin": ((B, K), torch.float32),
              "conf": ((B, K), torch.float32), "lse": ((B, K), torch.float32),
              "argmax": ((B, K), torch.int32), "k_next": ((B,), torch.int32),
              "n_accept": ((B,), torch.int32), "out_tokens": ((B, K), torch.int32),
              "accept": ((B, K), torch.uint8)}
    out, bufs = {}, {}
    for n, (shape, dt) in shapes.items():
        out[n], bufs[n] = _guarded(shape, dt)
    nws = cmsd.lib().cmsd_workspace_bytes(B, K, w.V)
    wsbuf = torch.full((nws + 4096,), 0xA5, dtype=torch.uint8, device="cuda")
    ws = wsbuf[:nws]
    ws.zero_()
    k_row = torch.tensor([7, 3, 0, 6, 1], dtype=torch.int32, device="cuda")
    p = cmsd.params(K, rule, **kw)
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    tok = torch.from_numpy(w.tokens).cuda()
    for it in range(3):
        cmsd.confidence_verify(d, t, tok, k_row=k_row, p=p, seed=w.seed, iteration=it, out=out, ws=ws)
    torch.cuda.synchronize()
    for n, (shape, dt) in shapes.items():
        assert _guards_intact(bufs[n], dt), n
    assert bool((wsbuf[nws:] == 0xA5).all().item()), "workspace overrun"
    g = {n: v.cpu().numpy() for n, v in out.items()}
    compare(w, g, oracle_fused(w, p, iteration=2, k_row=k_row.cpu().numpy()), k_row=k_row.cpu().numpy())


def test_device_error_word(cmsd, W):
    # drafted tokens outside [0, V) and k_row outside [0, K] are clamped on the
    # device before any load (token -> 0, k_row -> [0, K]) and reported in the
    # workspace error word: bit 0 and bit 1
    w = W.make("c2", B=4, K=5, V=900)
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    ws = cmsd.workspace(w.B, w.K, w.V)
    p = cmsd.params(w.K, "sampled")
    assert cmsd.workspace_errors(ws) == 0
    good = torch.from_numpy(w.tokens).cuda()
    cmsd.confidence_verify(d, t, good, p=p, ws=ws)
    assert cmsd.workspace_errors(ws) == 0
    bad = w.tokens.copy()
    bad[1, 2], bad[3, 0] = -1, w.V
    cmsd.confidence_verify(d, t, torch.from_numpy(bad).cuda(), p=p, ws=ws)
    assert cmsd.workspace_errors(ws) == 1
    assert cmsd.workspace_errors(ws) == 0                # reading clears the word
    kr = torch.tensor([5, 9, -2, 3], dtype=torch.int32, device="cuda")
    cmsd.confidence_verify(d, t, good, k_row=kr, p=p, ws=ws)
    assert cmsd.workspace_errors(ws) == 2
    cmsd.confidence_verify(d, t, torch.from_numpy(bad).cuda(), k_row=kr, p=p, ws=ws)
    assert cmsd.workspace_errors(ws) == 3
    # the workspace keeps working after errors: a clean call matches the oracle
    g = gpu_fused(cmsd, torch, w, p, iteration=2)
    compare(w, g, oracle_fused(w, p, iteration=2))


# ---------------------------------------------------------------- full sizes
#
# Every sequence of the full-size workloads, in the launch configuration
# bench.py times, against the oracle (run over the host's cores); flagged
# decisions bounded; deviations recorded (CMSD_PARITY_RECORD).

@pytest.fixture(scope="module")
def full_c3(W):
    return W.make("c3")


@pytest.fixture(scope="module")
def full_c4(W):
    return W.make("c4")


def _full_size(cmsd, w, name, rule, kw):
    import oracle_pool
    p = cmsd.params(w.K, rule, **kw)
    g = gpu_fused(cmsd, torch, w, p, iteration=1)
    check_properties(w, g, p)
    r = oracle_pool.fused(w, p.as_dict(), w.seed, iteration=1)
    f = compare(w, g, r)
    assert f["seqs"] == w.B and f["rows"] == w.B * w.K
    assert_flag_bound(f)
    record(name, rule, f, {"sizes": dict(B=w.B, K=w.K, V=w.V, dtype=w.dtype)})
    print(name, rule, f)


@pytest.mark.parametrize("rule,kw", RULES)
def test_full_size_c1_c2(cmsd, W, rule, kw):
    for name in ("c1", "c2"):
        _full_size(cmsd, W.make(name), name, rule, kw)


@pytest.mark.parametrize("rule,kw", RULES)
def test_full_size_c3(cmsd, full_c3, rule, kw):
    _full_size(cmsd, full_c3, "c3", rule, kw)


@pytest.mark.parametrize("rule,kw", RULES)
def test_full_size_c4(cmsd, full_c4, rule, kw):
    _full_size(cmsd, full_c4, "c4", rule, kw)


def _first_sequences(W, w, n):
    from paper_2508_15371_gb300.workloads import Workload
    return Workload(w.name, n, w.K, w.V, w.dtype, np.ascontiguousarray(w.draft[:n]),
                    np.ascontiguousarray(w.target[:n]), np.ascontiguousarray(w.tokens[:n]), w.seed)


@pytest.mark.parametrize("rule,kw", RULES)
@pytest.mark.parametrize("name,size,n", [
    ("c3", dict(B=64), (8, 1)),               # 7 warp pieces per row, then 57 and 62
    ("c2", dict(B=512, V=8192), (8, 1)),      # flat split over 4096 rows, then 4 pieces per row
])
def test_split_invariance(cmsd, W, name, size, n, rule, kw):
    # The merge of a row's per-warp partials does not depend on how the row is
    # cut: the same sequences inside a large batch and alone (different warp
    # splits) give the same signals to within fp32 reordering, the same argmax
    # and the same decisions (sequences the oracle flags as near a threshold
    # excepted).
    w = W.make(name, **size)
    p = cmsd.params(w.K, rule, **kw)
    big = gpu_fused(cmsd, torch, w, p, iteration=5)
    for m in n:
        ws = _first_sequences(W, w, m)
        small = gpu_fused(cmsd, torch, ws, p, iteration=5)
        r = oracle_fused(ws, p, iteration=5)
        for name_ in ("H", "margin", "conf", "lse"):
            d = np.abs(small[name_].astype(np.float64) - big[name_][:m])
            assert np.all(np.isfinite(small[name_]) == np.isfinite(big[name_][:m]))
            fin = np.isfinite(small[name_])
            assert d[fin].max(initial=0.0) <= 4e-6, (name_, m, float(d[fin].max()))
        assert np.array_equal(small["argmax"], big["argmax"][:m])
        for b in range(m):
            if r.k_flag[b] or r.n_flag[b] or r.tok_flag[b]:
                continue
            assert small["k_next"][b] == big["k_next"][b], (m, b)
            assert small["n_accept"][b] == big["n_accept"][b], (m, b)
            assert np.array_equal(small["out_tokens"][b], big["out_tokens"][b]), (m, b)


@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_max_window(cmsd, W, rule, kw):
    # K = 1024, the largest window: the epilogue takes the per-row path
    w = W.make("c2", B=2, K=1024, V=96, dtype="f32")
    p = cmsd.params(w.K, rule, **kw)
    compare(w, gpu_fused(cmsd, torch, w, p, iteration=2), oracle_fused(w, p, iteration=2))


@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_ragged_max_batch(cmsd, W, rule, kw):
    # B = 12000 sequences with a k_row (the largest ragged batch), windows of
    # 0..4 positions; every 97th sequence against the oracle, invariants on all
    import oracle_pool
    w = W.make("c2", B=12000, K=4, V=136, dtype="bf16")
    k_row = np.random.default_rng(12).integers(0, 5, w.B).astype(np.int32)
    p = cmsd.params(w.K, rule, **kw)
    g = gpu_fused(cmsd, torch, w, p, iteration=4, k_row=k_row)
    seqs = list(range(0, w.B, 97))
    r = oracle_pool.fused(w, p.as_dict(), w.seed, iteration=4, k_row=k_row, seqs=seqs)
    compare(w, g, r, k_row=k_row, seqs=seqs)
    n, k = g["n_accept"], g["k_next"]
    assert np.all((n >= 0) & (n <= k_row))
    assert np.all((k >= p.k_min) & (k <= p.k_max))
    for b in np.where(k_row == 0)[0]:
        assert n[b] == 0 and np.all(g["out_tokens"][b] == -1)


@pytest.mark.parametrize("rule,kw", RULES)
def test_parity_large_vocab(cmsd, W, rule, kw):
    # V = 1,000,003 (odd: unaligned rows, scalar heads and tails), about 127
    # warp pieces per row
    w = W.make("c2", B=1, K=3, V=1000003, dtype="f32")
    p = cmsd.params(w.K, rule, **kw)
    compare(w, gpu_fused(cmsd, torch, w, p, iteration=9), oracle_fused(w, p, iteration=9))
