"""Shared helpers of the GPU parity tests: run the library, run the oracle,
compare element by element with the documented tolerances, bound the number
of decisions the oracle flags as near a threshold, and record the largest
deviations."""
from __future__ import annotations

import json
import os

import numpy as np

import oracle as O

TOL = {"f32": 1e-5, "bf16": 2e-4}
# Decisions the oracle flags (within 1e-6 of a threshold) are excluded from
# the bit-exact checks; at most this fraction of a workload's decisions (and
# at least one) may be flagged, so that the exact checks are never vacuous.
FLAG_FRACTION = 0.005
SIGNALS = ("H", "margin", "conf", "lse")


def bonus_view(wp):
    """A workload drafted over K = wp.K - 1 positions whose verifier rows
    include the extra (bonus) row: drafter [B, K, V], target [B, K + 1, V]."""
    from paper_2508_15371_gb300.workloads import Workload
    K = wp.K - 1
    return Workload(wp.name + "+bonus", wp.B, K, wp.V, wp.dtype, np.ascontiguousarray(wp.draft[:, :K]),
                    wp.target, np.ascontiguousarray(wp.tokens[:, :K]), wp.seed)


def oracle_params(p):
    """oracle.Params from the library's cmsd_params (float32 values as float64)."""
    return O.Params(**p.as_dict())


def gpu_fused(cmsd, torch, w, p, seed=None, iteration=0, k_row=None):
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    tok = torch.from_numpy(np.ascontiguousarray(w.tokens)).cuda()
    kr = None if k_row is None else torch.from_numpy(np.asarray(k_row, np.int32)).cuda()
    out = cmsd.confidence_verify(d, t, tok, k_row=kr, p=p, seed=w.seed if seed is None else seed,
                                 iteration=iteration)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items() if v is not None}


def oracle_fused(w, p, seed=None, iteration=0, k_row=None, seqs=None):
    return O.confidence_verify(O.logits_to_f64(w.draft, w.dtype), O.logits_to_f64(w.target, w.dtype),
                               w.tokens, oracle_params(p), seed=w.seed if seed is None else seed,
                               iteration=iteration, k_row=k_row, seqs=seqs)


def compare(w, g, r, k_row=None, seqs=None, signals=True, report=None):
    """Assert parity of GPU outputs g (dict of numpy) with oracle result r.

    Floats within TOL[dtype]; argmax bit-exact; k_next, n_accept, out_tokens and
    accept bits bit-exact except where the oracle flags a near-threshold
    decision.  Returns a dict of flagged counts.
    """
    B, K = w.B, w.K
    kb = np.full(B, K) if k_row is None else np.asarray(k_row)
    seq_list = range(B) if seqs is None else seqs
    tol = TOL[w.dtype]
    flags = {"k": 0, "n": 0, "tok": 0, "acc": 0, "rows": 0, "seqs": 0}
    maxerr = {n: 0.0 for n in SIGNALS}
    for b in seq_list:
        k = int(kb[b])
        flags["seqs"] += 1
        flags["rows"] += k
        if signals and k:
            for name in SIGNALS:
                gv, rv = g[name][b, :k], getattr(r, name)[b, :k]
                fin = np.isfinite(rv)
                assert np.array_equal(np.isfinite(gv), fin), (name, b, gv, rv)
                err = np.abs(gv[fin].astype(np.float64) - rv[fin])
                assert err.size == 0 or err.max() <= tol, (name, b, float(err.max()), gv, rv)
                if err.size:
                    maxerr[name] = max(maxerr[name], float(err.max()))
            assert np.array_equal(g["argmax"][b, :k], r.argmax[b, :k]), ("argmax", b)
        if r.k_flag[b]:
            flags["k"] += 1
        elif "k_next" in g:
            assert g["k_next"][b] == r.k_next[b], ("k_next", b, g["k_next"][b], r.k_next[b])
        if r.n_accept is None:
            continue
        if r.n_flag[b]:
            flags["n"] += 1
        else:
            assert g["n_accept"][b] == r.n_accept[b], ("n_accept", b, g["n_accept"][b], r.n_accept[b])
        if r.tok_flag[b]:
            flags["tok"] += 1
        else:
            assert np.array_equal(g["out_tokens"][b], r.out_tokens[b]), \
                ("out_tokens", b, g["out_tokens"][b], r.out_tokens[b])
        if "accept" in g:
            for i in range(k):
                if r.acc_flag[b, i]:
                    flags["acc"] += 1
                else:
                    assert bool(g["accept"][b, i]) == bool(r.accept[b, i]), ("accept", b, i)
            assert not np.any(g["accept"][b, k:]), ("accept beyond k_row", b)
    if signals:
        flags["max_abs_err"] = maxerr
    if report is not None:
        report.append(flags)
    return flags


def flagged_total(flags):
    return flags["k"] + flags["n"] + flags["tok"] + flags["acc"]


def decisions_total(flags):
    """k_next, n_accept and correction token per sequence, accept bit per row."""
    return 3 * flags["seqs"] + flags["rows"]


def assert_flag_bound(flags):
    """The oracle flags at most FLAG_FRACTION of the decisions (at least one
    flag is always allowed): a bug that flagged everything would otherwise
    make every integer check vacuous."""
    nf, nd = flagged_total(flags), decisions_total(flags)
    assert nf <= max(1, FLAG_FRACTION * nd), (nf, nd, flags)


def record(name, rule, flags, extra=None):
    """Append one parity record to the JSON file named by CMSD_PARITY_RECORD
    (if set): flagged counts and the largest deviations of the signals."""
    path = os.environ.get("CMSD_PARITY_RECORD")
    if not path:
        return
    rec = {"workload": name, "rule": rule, "sequences": flags["seqs"], "rows": flags["rows"],
           "decisions": decisions_total(flags),
           "flagged": {k: flags[k] for k in ("k", "n", "tok", "acc")},
           "max_abs_err": flags.get("max_abs_err")}
    if extra:
        rec.update(extra)
    d = os.path.dirname(os.path.abspath(path))
    os.makedirs(d, exist_ok=True)
    with open(path, "a") as f:
        f.write(json.dumps(rec) + "\n")


def check_properties(w, g, p, k_row=None):
    """Properties that hold at any size (used where the oracle is not run)."""
    B, K, V = w.B, w.K, w.V
    kb = np.full(B, K) if k_row is None else np.asarray(k_row)
    kn = g["k_next"]
    assert np.all((kn >= p.k_min) & (kn <= p.k_max))
    n = g["n_accept"]
    assert np.all((n >= 0) & (n <= kb))
    ot = g["out_tokens"]
    for b in range(B):
        k, nb = int(kb[b]), int(n[b])
        assert np.array_equal(ot[b, :nb], w.tokens[b, :nb])
        if nb < k:
            assert 0 <= ot[b, nb] < V
            assert np.all(ot[b, nb + 1:] == -1)
        else:
            assert np.all(ot[b, k:] == -1)
        if "accept" in g:
            acc = g["accept"][b, :k].astype(bool)
            assert np.all(acc[:nb]) and (nb == k or not acc[nb])
    if "H" in g:
        H = g["H"][kb[:, None] > np.arange(K)[None, :]]
        assert np.all(H >= -1e-4) and np.all(H <= np.log(V) + 1e-3)
        c = g["conf"][kb[:, None] > np.arange(K)[None, :]]
        assert np.all((c >= 0) & (c <= 1))
