"""cmsd_confidence_verify_static (scratch in the library's device image, no
workspace) against cmsd_confidence_verify with a caller workspace.

Kept in a file of its own, collected last, so that it also runs after every
other GPU test in the same process; it must pass alone as well.
"""
import ctypes

import numpy as np
import pytest

from parity_util import TOL

pytestmark = pytest.mark.gpu

torch = pytest.importorskip("torch")

FLOATS = ("H", "margin", "conf", "lse")
INTS = ("argmax", "k_next", "n_accept", "out_tokens", "accept")


@pytest.fixture(scope="module")
def cmsd():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    from paper_2508_15371_gb300 import cmsd as c
    c.lib()
    return c


def _inputs(cmsd, name, **kw):
    from paper_2508_15371_gb300 import workloads
    w = workloads.make(name, **kw)
    d = cmsd.to_device_logits(w.draft, w.dtype)
    t = cmsd.to_device_logits(w.target, w.dtype)
    tok = torch.from_numpy(np.ascontiguousarray(w.tokens)).cuda()
    return w, d, t, tok


def _host(o):
    return {k: v.cpu().numpy() for k, v in o.items() if v is not None}


@pytest.mark.parametrize("name,kw,rule,k_row", [
    ("c2", dict(B=4, K=8, V=4096), "sampled", None),
    ("c2", dict(B=4, K=8, V=4096), "paper", None),
    ("c1", dict(B=3, K=5, V=2500), "sampled", [5, 2, 0]),
    ("c3", dict(B=2, K=8), "sampled", None),          # V = 128256
])
def test_static_scratch_matches_workspace_entry_point(cmsd, name, kw, rule, k_row):
    w, d, t, tok = _inputs(cmsd, name, **kw)
    kr = None if k_row is None else torch.tensor(k_row, dtype=torch.int32, device="cuda")
    p = cmsd.params(w.K, rule, beta_rank=0 if rule == "sampled" else 3)
    ref = _host(cmsd.confidence_verify(d, t, tok, k_row=kr, p=p, seed=w.seed, iteration=4))
    tol = TOL[w.dtype]
    kb = np.full(w.B, w.K) if k_row is None else np.asarray(k_row)
    for call in range(2):                    # two calls in a row on the same scratch
        got = _host(cmsd.confidence_verify_static(d, t, tok, k_row=kr, p=p, seed=w.seed, iteration=4))
        torch.cuda.synchronize()
        for b in range(w.B):
            k = int(kb[b])
            for n in FLOATS:
                a, r = got[n][b, :k], ref[n][b, :k]
                assert np.array_equal(np.isfinite(a), np.isfinite(r)), (call, n, b)
                fin = np.isfinite(r)
                assert np.all(np.abs(a[fin] - r[fin]) <= tol), (call, n, b, a, r)
            for n in ("argmax", "out_tokens", "accept"):
                assert np.array_equal(got[n][b, :k], ref[n][b, :k]), (call, n, b)
            assert np.array_equal(got["out_tokens"][b], ref["out_tokens"][b]), (call, b)
        assert np.array_equal(got["k_next"], ref["k_next"]), call
        assert np.array_equal(got["n_accept"], ref["n_accept"]), call


def test_static_scratch_rejects_oversize_problem(cmsd):
    # B*K = 131072 positions needs more than CMSD_STATIC_SCRATCH_BYTES; the call
    # is refused on the host after the argument checks and before anything is
    # enqueued (the aligned dummy pointers are never dereferenced)
    p = cmsd.params(1024, "sampled")
    a = ctypes.c_void_p(1 << 20)
    rc = cmsd.lib().cmsd_confidence_verify_static(
        a, a, a, None, 128, 1024, 32000, cmsd.BF16, ctypes.byref(p), 0, 0,
        None, None, None, None, None, None, a, a, None, None)
    assert rc == cmsd.ESCRATCH
    # an invalid argument is reported before the size limit
    rc = cmsd.lib().cmsd_confidence_verify_static(
        None, a, a, None, 128, 1024, 32000, cmsd.BF16, ctypes.byref(p), 0, 0,
        None, None, None, None, None, None, a, a, None, None)
    assert rc == cmsd.EINVAL
    assert b"static scratch" in cmsd.lib().cmsd_strerror(cmsd.ESCRATCH)
    # the empty problem is a valid call that enqueues nothing
    rc = cmsd.lib().cmsd_confidence_verify_static(
        None, None, None, None, 0, 8, 32000, cmsd.BF16, ctypes.byref(p), 0, 0,
        None, None, None, None, None, None, None, None, None, None)
    assert rc == cmsd.OK
