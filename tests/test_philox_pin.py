"""Pin the oracle's Philox4x32-10 to an independent implementation.

Triton ships its own Philox4x32 (triton.language.random.philox, ten rounds,
key = (seed low word, seed high word)); under TRITON_INTERPRET=1 it runs on
the CPU through numpy.  It is used here only as an outside reference for the
oracle's generator -- nothing in the library uses Triton.
"""
import json
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import scipy.stats as st

from oracle import philox

_PROBE = textwrap.dedent("""
    import json, os, sys
    os.environ["TRITON_INTERPRET"] = "1"
    import numpy as np, torch, triton, triton.language as tl

    @triton.jit
    def k(c_ptr, out_ptr, seed, n: tl.constexpr):
        o = tl.arange(0, n)
        c0 = tl.load(c_ptr + o * 4 + 0)
        c1 = tl.load(c_ptr + o * 4 + 1)
        c2 = tl.load(c_ptr + o * 4 + 2)
        c3 = tl.load(c_ptr + o * 4 + 3)
        a, b, c, d = tl.philox(seed, c0, c1, c2, c3)
        tl.store(out_ptr + o * 4 + 0, a)
        tl.store(out_ptr + o * 4 + 1, b)
        tl.store(out_ptr + o * 4 + 2, c)
        tl.store(out_ptr + o * 4 + 3, d)

    spec = json.loads(sys.stdin.read())
    res = {}
    for seed, ctrs in spec:
        n = len(ctrs)
        c = torch.tensor(np.array(ctrs, dtype=np.uint32).view(np.int32).reshape(-1))
        out = torch.zeros(4 * n, dtype=torch.int32)
        k[(1,)](c, out, seed, n)
        res[str(seed)] = out.numpy().view(np.uint32).reshape(n, 4).tolist()
    print(json.dumps(res))
""")


def _cases():
    rng = np.random.default_rng(2024)
    seeds = [0, 1, 4, 0xDEADBEEF, 0x123456789ABCDEF0]
    out = []
    for s in seeds:
        ctrs = [[0, 0, 0, 0], [0xFFFFFFFF] * 4, [1, 2, 3, 4]]
        ctrs += rng.integers(0, 2 ** 32, (13, 4), dtype=np.uint64).tolist()
        out.append((s, ctrs))
    return out


def test_philox_matches_triton_reference():
    pytest.importorskip("triton")
    pytest.importorskip("torch")
    cases = _cases()
    proc = subprocess.run([sys.executable, "-c", _PROBE], input=json.dumps(cases),
                          capture_output=True, text=True, timeout=600,
                          env=dict(os.environ, TRITON_INTERPRET="1"))
    if proc.returncode != 0:
        pytest.fail("triton interpreter probe failed:\n" + proc.stderr[-2000:])
    ref = json.loads(proc.stdout.strip().splitlines()[-1])
    for seed, ctrs in cases:
        key = philox.seed_key(seed)
        for ctr, want in zip(ctrs, ref[str(seed)]):
            assert list(philox.philox4x32_10(ctr, key)) == want
        c = np.array(ctrs, dtype=np.uint64)
        vec = philox.philox4x32_10_np(c[:, 0], c[:, 1], c[:, 2], c[:, 3], *key)
        assert np.stack(vec, axis=1).tolist() == ref[str(seed)]


def test_scalar_and_vector_forms_agree():
    rng = np.random.default_rng(1)
    c = rng.integers(0, 2 ** 32, (200, 4), dtype=np.uint64)
    key = philox.seed_key(987654321987)
    vec = np.stack(philox.philox4x32_10_np(c[:, 0], c[:, 1], c[:, 2], c[:, 3], *key), axis=1)
    for row, v in zip(c.tolist(), vec.tolist()):
        assert list(philox.philox4x32_10(row, key)) == v


def test_uniforms_are_uniform_and_distinct_streams():
    U = philox.residual_uniforms(5, 3, 2, 9, 200000)
    assert U.min() >= 0.0 and U.max() < 1.0
    assert st.kstest(U, "uniform").pvalue > 1e-3
    assert np.all(U * 2 ** 24 == np.floor(U * 2 ** 24))          # 24-bit grid
    U2 = philox.residual_uniforms(5, 3, 2, 10, 200000)
    assert st.pearsonr(U, U2)[0] < 0.01
    acc = np.array([philox.accept_uniform(0, b, i, it) for b in range(8) for i in range(8) for it in range(40)])
    assert st.kstest(acc, "uniform").pvalue > 1e-3
    # the acceptance, residual-entry and residual-group streams use different counters
    a0 = philox.accept_uniform(5, 3, 2, 9)
    assert a0 != U[0] or a0 != U[1]
    Ug = philox.group_uniforms(5, 3, 2, 9, 64)
    assert not np.array_equal(Ug[:8], U[:8])
    assert st.kstest(philox.group_uniforms(1, 0, 0, 3, 100000), "uniform").pvalue > 1e-3
