"""The residual draw by group bounds against the oracle.

Under the sampled rule without the bonus row the residual token is drawn by a
cluster of CTAs per rejected position: the target row's group maxima bound
each group's residual mass, and only the groups that bound cannot rule out
are raced exactly (the same keys as the race over every group, so the same
token; Sec. III.B(c) residual, drawn by the two-level exponential race).
These cases aim at the paths that choice opens: candidate lists that
overflow (flat rows), empty and near-empty residuals, target groups masked
to -inf, rows off 16-byte boundaries, row shares that are empty, more queued
rows than clusters, and the largest share that fits shared memory next to
the first that does not (which takes the race over every group).  Tokens,
accepted lengths and the rest are compared element by element
(parity_util.compare).
"""
import numpy as np
import pytest

from parity_util import compare, gpu_fused, oracle_fused
from paper_2508_15371_gb300 import workloads as W

pytestmark = pytest.mark.gpu
torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def cmsd():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2508_15371_gb300 import cmsd as c
    c.lib()
    return c


def _wl(d, t, tok, dtype, seed=5, name="bounds"):
    B, K, V = d.shape
    if dtype == "bf16":
        d, t = W.f32_to_bf16_bits(d), W.f32_to_bf16_bits(t)
    return W.Workload(name=name, B=B, K=K, V=V, dtype=dtype, draft=d, target=t,
                      tokens=np.ascontiguousarray(tok, dtype=np.int32), seed=seed)


def _synthetic(rng, B, K, V, sd, noise):
    d = rng.normal(0, sd, (B, K, V)).astype(np.float32)
    t = (d + rng.normal(0, noise, (B, K, V))).astype(np.float32) if noise > 0 else d.copy()
    return d, t, rng.integers(0, V, (B, K)).astype(np.int32)


def _check(cmsd, w, iterations, tau=0.1, min_rejected=1):
    p = cmsd.params(w.K, "sampled", beta_rank=0, tau_base=tau)
    rejected = 0
    for it in iterations:
        g = gpu_fused(cmsd, torch, w, p, iteration=it)
        compare(w, g, oracle_fused(w, p, iteration=it))
        rejected += int((g["n_accept"] < w.K).sum())
    assert rejected >= min_rejected
    return rejected


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_flat_rows_overflow_the_candidate_list(cmsd, dtype):
    # nearly uniform rows: every group's bound is close to its mass, thousands
    # of groups stay candidates and each CTA races its whole share
    rng = np.random.default_rng(1)
    _check(cmsd, _wl(*_synthetic(rng, 6, 4, 65536, sd=0.02, noise=0.02), dtype), range(3), tau=-3.0)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_target_equal_to_drafter(cmsd, dtype):
    # p and q differ by rounding only: near-empty residuals, and empty ones
    # that fall back to the target argmax
    rng = np.random.default_rng(2)
    _check(cmsd, _wl(*_synthetic(rng, 8, 4, 8192, sd=2.0, noise=0.0), dtype), range(3), tau=-5.0)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_masked_target_groups(cmsd, dtype):
    # whole groups and single entries of the target at -inf (p = 0 there), a
    # peaked drafter elsewhere
    rng = np.random.default_rng(3)
    B, K, V = 8, 4, 16384
    d = rng.normal(0, 1.0, (B, K, V)).astype(np.float32)
    d[:, :, rng.integers(0, V, 8)] += 8.0
    t = (d + rng.normal(0, 1.0, (B, K, V))).astype(np.float32)
    grp = rng.random((B, K, V // 32)) < 0.5
    t.reshape(B, K, V // 32, 32)[grp] = -np.inf
    t[rng.random((B, K, V)) < 0.1] = -np.inf
    t[:, :, 0] = 0.0                                   # every row keeps a finite entry
    tok = rng.integers(0, V, (B, K)).astype(np.int32)
    _check(cmsd, _wl(d, t, tok, dtype), range(4))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("V", [2, 33, 100, 4097])
def test_tiny_and_odd_vocabularies(cmsd, dtype, V):
    # shares of one group or none; rows off 16-byte boundaries (element loads)
    rng = np.random.default_rng(V)
    _check(cmsd, _wl(*_synthetic(rng, 6, 3, V, sd=1.5, noise=1.0), dtype), range(4), tau=-1.0)


def test_more_rows_than_clusters(cmsd):
    # 600 sequences, one position each: the clusters loop over the queued rows
    rng = np.random.default_rng(6)
    assert _check(cmsd, _wl(*_synthetic(rng, 600, 1, 2048, sd=1.0, noise=1.5), "bf16"), range(1),
                  tau=-1.0) > 304


@pytest.mark.parametrize("V", [152064, 200000])
def test_largest_shares(cmsd, V):
    # f32 rows: 152064 entries fill most of the CTA's shared memory; 200000 do
    # not fit and take the race over every group
    rng = np.random.default_rng(7)
    _check(cmsd, _wl(*_synthetic(rng, 2, 2, V, sd=2.0, noise=1.0), "f32"), range(3), tau=-1.0)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_rows_at_16_byte_offsets(cmsd, dtype):
    # logits at a base 16 bytes past an allocation's start
    rng = np.random.default_rng(8)
    w = _wl(*_synthetic(rng, 5, 6, 12800, sd=1.5, noise=1.0), dtype)
    p = cmsd.params(w.K, "sampled", beta_rank=0, tau_base=-1.0)
    shift = 16 // (4 if dtype == "f32" else 2)

    def shifted(x):
        buf = torch.empty(x.numel() + shift, dtype=x.dtype, device=x.device)
        y = buf[shift:].view(x.shape)
        y.copy_(x)
        return y

    d = shifted(cmsd.to_device_logits(w.draft, w.dtype))
    t = shifted(cmsd.to_device_logits(w.target, w.dtype))
    tok = torch.from_numpy(w.tokens).cuda()
    for it in range(3):
        o = cmsd.confidence_verify(d, t, tok, p=p, seed=w.seed, iteration=it)
        g = {k: v.cpu().numpy() for k, v in o.items() if v is not None}
        compare(w, g, oracle_fused(w, p, iteration=it))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_decisions_without_signal_outputs(cmsd, dtype):
    # Without the per-position signals the pass does not re-read the vectors
    # holding the maxima. Each lane's vector start then stands in for the
    # argmax index in the merges. Drafter rows whose maximum value repeats
    # check that the second-largest logit still sees the repeat (margin 0):
    # - in the same 16-byte vector;
    # - 64 entries on (another lane);
    # - half a row on (another warp).
    rng = np.random.default_rng(9)
    B, K, V = 8, 6, 40000
    d, t, tok = _synthetic(rng, B, K, V, sd=1.5, noise=1.0)
    for b in range(B):
        for i in range(K):
            j = int(np.argmax(d[b, i]))
            for off in ((1, 64, V // 2), (1,), (64,), (V // 2,), ())[(b + i) % 5]:
                d[b, i, (j + off) % V] = d[b, i, j]
    w = _wl(d, t, tok, dtype)
    p = cmsd.params(K, "sampled", beta_rank=0, tau_base=0.0)
    dd = cmsd.to_device_logits(w.draft, w.dtype)
    tt = cmsd.to_device_logits(w.target, w.dtype)
    tk = torch.from_numpy(w.tokens).cuda()
    for it in range(3):
        full = gpu_fused(cmsd, torch, w, p, iteration=it)
        compare(w, full, oracle_fused(w, p, iteration=it))
        o = cmsd.confidence_verify(dd, tt, tk, p=p, seed=w.seed, iteration=it, signals=False)
        for k in ("n_accept", "out_tokens", "k_next"):
            assert np.array_equal(o[k].cpu().numpy(), full[k]), k


def test_record_wait_runs_out(cmsd):
    # The draw launched alone, with no streaming pass to release the records:
    # - each sequence's bounded wait gives up after about a second;
    # - the draw sets error bit 2 and writes no token;
    # - the context and the workspace then serve an ordinary call.
    import time
    rng = np.random.default_rng(10)
    w = _wl(*_synthetic(rng, 4, 3, 4096, sd=1.0, noise=1.0), "bf16")
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    ws = cmsd.workspace(w.B, w.K, w.V)
    out = torch.full((w.B, w.K), 7, dtype=torch.int32, device="cuda")
    cmsd.workspace_errors(ws)
    t0 = time.perf_counter()
    rc = cmsd.lib().cmsd_test_record_wait_timeout(cmsd._ptr(d), cmsd._ptr(t), w.B, w.K, w.V, cmsd.BF16,
                                                  cmsd._ptr(out), cmsd._ptr(ws), ws.numel(), cmsd._stream())
    assert rc == cmsd.OK
    torch.cuda.synchronize()
    assert 0.5 < time.perf_counter() - t0 < 60
    assert cmsd.workspace_errors(ws) & 4
    assert bool((out == 7).all().item())
    p = cmsd.params(w.K, "sampled", beta_rank=0, tau_base=-1.0)
    compare(w, gpu_fused(cmsd, torch, w, p, iteration=1), oracle_fused(w, p, iteration=1))
    assert cmsd.workspace_errors(ws) == 0
