"""The C-ABI library without a GPU: it loads, exports every symbol the headers
declare, computes Philox on the host like the oracle, and rejects bad
arguments on the host before touching CUDA."""
import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PKG = os.path.join(ROOT, "paper_2508_15371_gb300")


def _built(name):
    path = os.path.join(PKG, name)
    if not os.path.exists(path):
        from paper_2508_15371_gb300 import build
        build.build()
    return path


def _declared(header):
    src = open(os.path.join(ROOT, "include", header)).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(cmsd_\w+)\s*\(", src)))


@pytest.mark.parametrize("header,lib", [("cmsd.h", "libcmsd.so"), ("cmsd_workload.h", "libcmsd_workload.so")])
def test_library_exports_every_declared_symbol(header, lib):
    L = ctypes.CDLL(_built(lib))
    names = _declared(header)
    assert names
    for n in names:
        assert hasattr(L, n), f"{lib} does not export {n}"


@pytest.fixture(scope="module")
def cmsd():
    _built("libcmsd.so")
    from paper_2508_15371_gb300 import cmsd as c
    c.lib()
    return c


def test_host_philox_matches_oracle(cmsd):
    from oracle import philox
    rng = np.random.default_rng(3)
    for _ in range(300):
        seed = int(rng.integers(0, 2 ** 63))
        c = [int(x) for x in rng.integers(0, 2 ** 32, 4)]
        want = philox.philox4x32_10(c, philox.seed_key(seed))
        for wd in range(4):
            assert cmsd.philox_u32(seed, *c, wd) == want[wd]


def test_params_default(cmsd):
    p = cmsd.params(8, "paper")
    assert (p.k_min, p.k_max, p.beta_rank, p.tau_sign, p.rule) == (1, 8, 3, 1, 0)
    assert abs(p.tau_base - 0.1) < 1e-7 and abs(sum(p.lam) - 1) < 1e-6
    s = cmsd.params(16, "sampled")
    assert (s.k_max, s.beta_rank, s.rule) == (16, 0, 1)


def _call_conf(cmsd, draft=8192, B=2, K=4, V=100, dtype=1, p=None):
    p = p if p is not None else cmsd.params(K)
    L = cmsd.lib()
    return L.cmsd_confidence(ctypes.c_void_p(draft) if draft else None, B, K, V, dtype, None,
                             ctypes.byref(p) if p is not False else None,
                             None, None, None, None, None, None, None, 0, None)


def test_argument_errors_rejected_on_host(cmsd):
    assert _call_conf(cmsd, B=0) == cmsd.OK                 # empty call: nothing to do
    assert _call_conf(cmsd, K=0) == cmsd.OK
    assert _call_conf(cmsd, V=1) == cmsd.EINVAL
    assert _call_conf(cmsd, B=-1) == cmsd.EINVAL
    assert _call_conf(cmsd, K=2000) == cmsd.EINVAL
    assert _call_conf(cmsd, dtype=7) == cmsd.EDTYPE
    assert _call_conf(cmsd, draft=0) == cmsd.EINVAL
    assert _call_conf(cmsd, draft=8200) == cmsd.EALIGN
    assert _call_conf(cmsd, p=False) == cmsd.EINVAL
    assert _call_conf(cmsd, B=1 << 20, K=1024, V=1 << 20) == cmsd.EINVAL   # B*K*V >= 2^46
    for bad in (dict(k_min=0), dict(k_min=5, k_max=4), dict(lam=(0.5, 0.5, 0.5)),
                dict(lam=(1.2, -0.1, -0.1)), dict(beta_sig=0.0), dict(alpha=0.0),
                dict(alpha=1.5), dict(beta_rank=-1), dict(tau_sign=0), dict(tau_base=float("inf"))):
        assert _call_conf(cmsd, p=cmsd.params(4, **bad)) == cmsd.EINVAL, bad


def test_verify_argument_errors(cmsd):
    L = cmsd.lib()
    p = cmsd.params(4, "sampled")
    a = ctypes.c_void_p(4096)
    # sampled rule needs draft_lse
    rc = L.cmsd_verify(a, a, a, None, 2, 4, 100, 1, ctypes.byref(p), a, None, 0, 0, a, a, None,
                       None, 0, None)
    assert rc == cmsd.EINVAL
    p.rule = 5
    rc = L.cmsd_verify(a, a, a, None, 2, 4, 100, 1, ctypes.byref(p), a, a, 0, 0, a, a, None,
                       None, 0, None)
    assert rc == cmsd.EDTYPE
    q = cmsd.params(4, "paper")
    rc = L.cmsd_confidence_verify(a, ctypes.c_void_p(4100), a, None, 2, 4, 100, 1, ctypes.byref(q), 0, 0,
                                  None, None, None, None, None, None, a, a, None, None, 0, None)
    assert rc == cmsd.EALIGN
    rc = L.cmsd_confidence_verify(a, a, a, None, 2, 4, 100, 1, ctypes.byref(q), 0, 0,
                                  None, None, None, None, None, None, None, a, None, None, 0, None)
    assert rc == cmsd.EINVAL          # n_accept is required
    assert L.cmsd_strerror(cmsd.ENOWS).decode().startswith("workspace")


def test_product_path_fails_loudly_without_library(tmp_path, monkeypatch):
    from paper_2508_15371_gb300 import cmsd as c
    monkeypatch.setattr(c, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(c, "_lib", None)
    with pytest.raises(c.CmsdError):
        c.lib()


def test_ablation_presets(cmsd):
    # the variants of the ablation (Sec. IV, Table III) as parameter sets
    full = cmsd.params(16, "sampled")
    assert (full.k_fixed, full.bonus) == (0, 0)
    fk = cmsd.params(16, "sampled", preset="fixed_k")
    assert fk.k_fixed == 16 and abs(fk.gamma - 1.0) < 1e-7
    ft = cmsd.params(16, "sampled", preset="fixed_tau")
    assert ft.k_fixed == 0 and ft.gamma == 0.0
    fkt = cmsd.params(16, "sampled", preset="fixed_k_tau")
    assert fkt.k_fixed == 16 and fkt.gamma == 0.0
    for name, j in (("entropy_only", 0), ("margin_only", 1), ("softmax_only", 2)):
        q = cmsd.params(16, "paper", preset=name)
        assert list(q.lam) == [1.0 if k == j else 0.0 for k in range(3)]
    p = cmsd.Params()
    assert cmsd.lib().cmsd_params_preset(ctypes.byref(p), 8, 0, 99) == cmsd.EINVAL


def test_bonus_and_fixed_k_argument_checks(cmsd):
    # k_fixed outside [k_min, k_max] and a bonus row with rows that are not a
    # whole number of 16-byte vectors are refused on the host
    L = cmsd.lib()
    a = ctypes.c_void_p(1 << 20)
    bad_k = cmsd.params(8, "paper", k_fixed=9)
    rc = L.cmsd_confidence_verify(a, a, a, None, 2, 8, 4096, cmsd.BF16, ctypes.byref(bad_k), 0, 0,
                                  None, None, None, None, None, None, a, a, None, None, 0, None)
    assert rc == cmsd.EINVAL
    odd = cmsd.params(8, "paper", bonus=1)
    rc = L.cmsd_confidence_verify(a, a, a, None, 2, 8, 4097, cmsd.BF16, ctypes.byref(odd), 0, 0,
                                  None, None, None, None, None, None, a, a, None, None, 0, None)
    assert rc == cmsd.EINVAL
