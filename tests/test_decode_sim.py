"""Decode-loop simulation (Algorithm 1 as a control loop over synthetic logits).

The device generator must reproduce the host recipe bit for bit, and the
simulated loop (k_next fed back as the next k_row on the device) must follow
the oracle's replay of the same sequences: k, n_accept and output tokens per
iteration, up to the first iteration where the oracle flags a decision at a
threshold (later iterations depend on that float-order tie).
"""
import numpy as np
import pytest

from parity_util import oracle_params

torch = pytest.importorskip("torch")


@pytest.fixture(scope="module")
def mods():
    from paper_2508_15371_gb300 import cmsd, decode_sim, workloads
    return cmsd, decode_sim, workloads


def test_summarize_counts(mods):
    _, ds, _ = mods
    hist = {"k": np.array([[4, 4], [2, 4]]), "n_accept": np.array([[4, 1], [0, 4]])}
    s = ds.summarize(hist)
    assert s["rollbacks"] == 2 and s["rows"] == 14
    assert s["mean_accepted"] == pytest.approx(9 / 4)
    assert s["tokens_per_iteration"] == pytest.approx((4 + 2 + 1 + 4) / 4)
    sb = ds.summarize(hist, bonus=True)          # a fully accepted window adds the verifier's token
    assert sb["tokens_per_iteration"] == pytest.approx((5 + 2 + 1 + 5) / 4)
    # pass bytes: drafted row pairs, bonus rows, rejected row pairs again
    assert ds.pass_bytes(hist, 10, 4) == (14 * 2 + 2 * 2) * 10 * 4
    assert ds.pass_bytes(hist, 10, 4, bonus=True) == (14 * 2 + 4 + 2 * 2) * 10 * 4


@pytest.mark.gpu
@pytest.mark.parametrize("bonus", [0, 1])
@pytest.mark.parametrize("V,k_row", [(1000, [5, 2, 0]), (4099, [1, 5, 3])])
def test_device_generator_matches_host(mods, V, k_row, bonus):
    cmsd, ds, W = mods
    assert torch.cuda.is_available()
    B, K = 3, 5
    p = cmsd.params(K, bonus=bonus)
    sim = ds.DecodeSim(B, K, V, 3, p, seed=4)
    table = W.normal_table()
    heights = W.ar1_heights(B, 3, 4, table)
    for it in (0, 2):
        sim.hist_k[it] = torch.tensor(k_row, dtype=torch.int32, device="cuda")
        sim.generate(it)
        torch.cuda.synchronize()
        d, t, tok = sim.draft.cpu().numpy(), sim.target.cpu().numpy(), sim.tokens.cpu().numpy()
        for b in range(B):
            hd, ht, htok = W.decode_iteration_host(table, heights, it, b, k_row[b], K, V, 4, bonus=bool(bonus))
            assert ht.shape[0] == k_row[b] + bonus
            for i in range(k_row[b]):
                assert np.array_equal(d[b, i].view(np.uint32), hd[i].view(np.uint32)), (it, b, i)
                assert tok[b, i] == htok[i], (it, b, i)
            for i in range(k_row[b] + bonus):
                assert np.array_equal(t[b, i].view(np.uint32), ht[i].view(np.uint32)), (it, b, i)


def _compare_with_oracle(cmsd, ds, W, B, K, V, iterations, rule, seqs, graph=False, **kw):
    import oracle as O
    p = cmsd.params(K, rule, beta_rank=0 if rule == "sampled" else 3, **kw)
    sim = ds.DecodeSim(B, K, V, iterations, p, seed=4)
    hist = sim.run(graph=graph)
    table = W.normal_table()
    heights = W.ar1_heights(B, iterations, 4, table)

    def gen(it, b, k):
        return W.decode_iteration_host(table, heights, it, b, k, K, V, 4, bonus=bool(p.bonus))

    compared = 0
    for b in seqs:
        traj = O.decode_sim_sequence(gen, b, iterations, K, oracle_params(p), 4)
        for it, st in enumerate(traj):
            assert hist["k"][it, b] == st["k"], (rule, b, it)
            if st["flagged"]:
                break
            assert hist["n_accept"][it, b] == st["n_accept"], (rule, b, it)
            assert np.array_equal(hist["out_tokens"][it, b], st["out_tokens"]), (rule, b, it)
            compared += 1
    return hist, compared


@pytest.mark.gpu
@pytest.mark.parametrize("graph", [False, True])
@pytest.mark.parametrize("rule", ["paper", "sampled"])
def test_decode_loop_matches_oracle(mods, rule, graph):
    cmsd, ds, W = mods
    hist, compared = _compare_with_oracle(cmsd, ds, W, 4, 16, 2048, 10, rule, range(4), graph=graph)
    assert compared >= 20
    k, n = hist["k"], hist["n_accept"]
    assert np.all((k >= 1) & (k <= 16)) and np.all((n >= 0) & (n <= k))


@pytest.mark.gpu
@pytest.mark.parametrize("rule", ["paper", "sampled"])
@pytest.mark.parametrize("preset,kw", [("full", dict(bonus=1)), ("fixed_k", {}), ("fixed_tau", {}),
                                       ("entropy_only", {})])
def test_decode_loop_variants_match_oracle(mods, rule, preset, kw):
    # the ablation variants and the bonus row, through the loop (CUDA graph)
    cmsd, ds, W = mods
    hist, compared = _compare_with_oracle(cmsd, ds, W, 3, 8, 1024, 8, rule, range(3), graph=True,
                                          preset=preset, **kw)
    assert compared >= 12
    s = ds.summarize(hist, bonus=bool(kw.get("bonus")))
    assert 0 < s["tokens_per_iteration"] <= 9


@pytest.mark.gpu
@pytest.mark.parametrize("rule", ["sampled", "paper"])
def test_decode_loop_full_size(mods, rule):
    # B=32, K_max=16, V=32000 float32 logits, 512 iterations: every sequence
    # against the oracle's replay (over the host's cores) up to its first
    # flagged iteration, invariants everywhere
    import oracle_pool
    from parity_util import record
    cmsd, ds, W = mods
    B, K, V, its = 32, 16, 32000, 512
    p = cmsd.params(K, rule, beta_rank=0 if rule == "sampled" else 3)
    sim = ds.DecodeSim(B, K, V, its, p, seed=4)
    hist = sim.run(graph=True)
    k, n, toks = hist["k"], hist["n_accept"], hist["out_tokens"]
    assert np.all((k >= 1) & (k <= K)) and np.all((n >= 0) & (n <= k))
    for it in range(its):
        for b in range(B):
            kk, nn = k[it, b], n[it, b]
            assert np.all(toks[it, b, kk:] == -1)
            assert np.all((toks[it, b, :min(nn + 1, kk)] >= 0) & (toks[it, b, :min(nn + 1, kk)] < V))
    s = ds.summarize(hist)
    assert s["rows"] == int(k.sum()) and 0 < s["mean_accepted"] <= K

    replays = oracle_pool.decode_replays(B, K, V, its, p.as_dict(), 4, range(B))
    compared, stopped = 0, []
    for b in range(B):
        for it, st in enumerate(replays[b]):
            assert k[it, b] == st["k"], (b, it)
            if st["flagged"]:
                stopped.append(it)
                break
            assert n[it, b] == st["n_accept"], (b, it)
            assert np.array_equal(toks[it, b], st["out_tokens"]), (b, it)
            compared += 1
    # the comparison covers (nearly) the whole trajectory of every sequence
    assert compared >= 0.9 * B * its, (compared, stopped)
    record("c5", rule, {"seqs": B, "rows": int(k.sum()), "k": 0, "n": 0, "tok": 0, "acc": 0},
           {"iterations_compared": compared, "iterations_total": B * its,
            "sequences_stopped_at_a_flagged_iteration": len(stopped),
            "first_flagged_iterations": sorted(stopped), "summary": s})
