"""GPU parity of the fused LM head + confidence entry point
(cmsd_lmhead_confidence) against the oracle (oracle/lmhead.py).

Two input recipes (paper_2508_15371_gb300/workloads.make_lmhead):
  exact      entries are multiples of 1/16, so every partial sum of every dot
             product is exact in fp32: the kernel's logits must equal the
             float64 logits bit for bit, the argmax must match exactly (ties
             to the lowest index included), and the signals must agree within
             the fp32-logit tolerance of the logits pass (1e-5).
  realistic  normal weights and spiked hidden states: each logit may differ
             from the exact dot product by fp32 rounding, at most
             d 2^-23 sum_j |h_j w_vj| (a sum of d terms, each addition off by
             at most one ulp of the running sum); the signals may then move by
             the first-order bounds of oracle.signal_error_bound, plus 1e-5.
"""
import numpy as np
import pytest

import oracle as O
from paper_2508_15371_gb300 import workloads as W

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

TOL = 1e-5


@pytest.fixture(scope="module")
def cmsd():
    from paper_2508_15371_gb300 import cmsd as C
    assert torch.cuda.is_available()
    return C


def _dev(bits):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda()


def _run(cmsd, w, P, logits=True):
    out = cmsd.lmhead_confidence(_dev(w.hidden), _dev(w.weight), p=P, logits=logits)
    torch.cuda.synchronize()
    return {k: v.cpu().numpy() for k, v in out.items()}


def _params(cmsd, **kw):
    p = cmsd.params(1, **kw)
    P = O.Params(lam=tuple(p.lam), beta_sig=p.beta_sig)
    return p, P


# R picks the hidden-row block: 64 (R <= 64), 128 (R <= 128), 256 (more; R > 256 takes several blocks)
@pytest.mark.parametrize("R,d,V", [(5, 256, 1000), (3, 64, 1003), (1, 128, 2), (64, 512, 4096), (7, 192, 129),
                                   (65, 128, 3000), (128, 256, 2049), (130, 128, 5000), (256, 64, 1500),
                                   (300, 128, 777)])
def test_exact_inputs_bit_exact(cmsd, R, d, V):
    w = W.make_lmhead(R=R, d=d, V=V, seed=R + d + V, exact=True)
    p, P = _params(cmsd)
    g = _run(cmsd, w, p)
    o = O.lm_head_confidence(w.hidden, w.weight, P)
    assert np.array_equal(g["logits"].astype(np.float64), o["logits"])
    assert np.array_equal(g["argmax"], o["argmax"])
    for k in ("H", "margin", "lse", "conf"):
        assert np.max(np.abs(g[k] - o[k])) <= TOL, k


@pytest.mark.parametrize("R,d,V", [(64, 512, 20000), (16, 1024, 32000)])
def test_realistic_inputs_within_rounding_bounds(cmsd, R, d, V):
    w = W.make_lmhead(R=R, d=d, V=V, seed=11)
    p, P = _params(cmsd)
    g = _run(cmsd, w, p)
    o = O.lm_head_confidence(w.hidden, w.weight, P)
    h = np.abs(O.bf16_bits_to_f64(w.hidden))
    ww = np.abs(O.bf16_bits_to_f64(w.weight))
    bound = d * 2.0 ** -23 * (h @ ww.T)                 # per logit
    err = np.abs(g["logits"].astype(np.float64) - o["logits"])
    assert np.all(err <= bound)
    eps = bound.max(axis=1)
    for r in range(R):
        b = O.signal_error_bound(eps[r], o["H"][r], V, P.lam, P.beta_sig)
        assert abs(g["lse"][r] - o["lse"][r]) <= b["lse"] + TOL
        assert abs(g["H"][r] - o["H"][r]) <= b["H"] + TOL
        assert abs(g["conf"][r] - o["conf"][r]) <= b["conf"] + TOL
        if o["margin"][r] > 2 * eps[r]:                  # the argmax cannot flip
            assert g["argmax"][r] == o["argmax"][r]
            assert abs(g["margin"][r] - o["margin"][r]) <= b["margin"] + TOL


def test_without_logits_output_same_signals(cmsd):
    w = W.make_lmhead(R=9, d=256, V=3000, seed=3, exact=True)
    p, _ = _params(cmsd)
    a = _run(cmsd, w, p, logits=True)
    b = _run(cmsd, w, p, logits=False)
    for k in ("H", "margin", "argmax", "conf", "lse"):
        assert np.array_equal(a[k], b[k]), k


def test_full_size_exact_sampled_rows(cmsd):
    # a 1B-class drafter head at a Llama-3 vocabulary, 64 rows; the oracle on 8 of them
    R, d, V = 64, 2048, 128256
    w = W.make_lmhead(R=R, d=d, V=V, seed=7, exact=True)
    p, P = _params(cmsd)
    g = _run(cmsd, w, p, logits=False)
    rows = np.arange(0, R, 8)
    o = O.lm_head_confidence(w.hidden[rows], w.weight, P)
    assert np.array_equal(g["argmax"][rows], o["argmax"])
    for k in ("H", "margin", "lse", "conf"):
        assert np.max(np.abs(g[k][rows] - o[k])) <= TOL, k
    # every row: the properties that hold at any size
    assert np.all((g["argmax"] >= 0) & (g["argmax"] < V))
    assert np.all((g["H"] >= -TOL) & (g["H"] <= np.log(V) + TOL))
    assert np.all((g["conf"] >= 0) & (g["conf"] <= 1)) and np.all(g["margin"] >= 0)


def test_argument_errors(cmsd):
    L = cmsd.lib()
    import ctypes
    p = cmsd.params(1)
    x = torch.zeros((4, 64), dtype=torch.int16, device="cuda")
    ws = cmsd.lmhead_workspace(4, 64, 4)
    args = lambda R, d, V, h, wt, wsz: (cmsd._ptr(h), cmsd._ptr(wt), R, d, V, ctypes.byref(p), None, None, None,
                                        None, None, None, cmsd._ptr(ws), wsz, cmsd._stream())
    assert L.cmsd_lmhead_confidence(*args(4, 63, 4, x, x, ws.numel())) == cmsd.EINVAL
    assert L.cmsd_lmhead_confidence(*args(4, 64, 1, x, x, ws.numel())) == cmsd.EINVAL
    assert L.cmsd_lmhead_confidence(*args(4, 64, 4, None, x, ws.numel())) == cmsd.EINVAL
    assert L.cmsd_lmhead_confidence(*args(4, 64, 4, x, x, 16)) == cmsd.ENOWS
    off = torch.zeros(4 * 64 + 8, dtype=torch.int16, device="cuda")[1:]
    assert L.cmsd_lmhead_confidence(*args(4, 64, 4, off, x, ws.numel())) == cmsd.EALIGN
    assert L.cmsd_lmhead_confidence(*args(0, 64, 4, x, x, ws.numel())) == cmsd.OK
