"""Algorithm 1 as a control loop over synthetic logits (decode-loop simulation).

The paper's drafter and verifier models (Sec. IV.A) are not available, so their
logits are produced on the device by libcmsd_workload.so, bit-identical to the
host recipe in workloads.py (decode_row_host: a drafter row with one spike
whose height drifts per sequence as an AR(1) process, and a noisy verifier).

Each iteration drafts k_row[b] positions of every sequence b, runs the fused
pass of libcmsd.so with that k_row, and the k_next it returns is the next
iteration's k_row (Sec. III.B(b)): the call writes it straight into the next
row of the k history, so the loop keeps no state on the host and needs no
copies -- per iteration one generator launch and the pass's one or two
kernels.  The whole loop can be captured once into a CUDA graph and replayed.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

from . import cmsd, workloads

_PKG = os.path.dirname(os.path.abspath(__file__))
WORKLOAD_LIB_PATH = os.path.join(_PKG, "libcmsd_workload.so")

_wlib = None
_wlib_lock = threading.Lock()


def wlib():
    """The loaded libcmsd_workload.so (raises if it is missing)."""
    global _wlib
    if _wlib is None:
        with _wlib_lock:
            if _wlib is None:
                if not os.path.exists(WORKLOAD_LIB_PATH):
                    raise cmsd.CmsdError(f"{WORKLOAD_LIB_PATH} is missing: build it with "
                                         "`python -c 'import __graft_entry__ as g; g.build()'`")
                L = ctypes.CDLL(WORKLOAD_LIB_PATH)
                vp = ctypes.c_void_p
                L.cmsd_gen_decode_rows.restype = ctypes.c_int
                L.cmsd_gen_decode_rows.argtypes = [vp, vp, ctypes.c_uint32, ctypes.c_int, ctypes.c_int,
                                                   ctypes.c_int, ctypes.c_int, vp, ctypes.c_uint64, vp, vp,
                                                   vp, vp]
                _wlib = L
    return _wlib


class DecodeSim:
    """State of one simulated decode loop: B sequences, window K_max, V logits.

    `p` is a cmsd.Params (its bonus flag adds the verifier's extra row);
    `seed` keys both the logit generator and the method's own uniforms.
    History on the device: hist_k[it] is the window drafted at iteration it
    (hist_k[0] = K_max, hist_k[it + 1] = k_next of iteration it), hist_n and
    hist_tok the accepted lengths and emitted tokens.
    """

    def __init__(self, B, K_max, V, iterations, p, seed=4, device="cuda"):
        import torch
        self.B, self.K_max, self.V, self.iterations = int(B), int(K_max), int(V), int(iterations)
        self.p, self.seed = p, int(seed)
        self.Kt = self.K_max + 1 if p.bonus else self.K_max
        dev = torch.device(device)
        self.table = torch.from_numpy(workloads.normal_table()).to(dev)
        self.heights = torch.from_numpy(workloads.ar1_heights(self.B, self.iterations, self.seed,
                                                              workloads.normal_table())).to(dev)
        self.draft = torch.zeros((self.B, self.K_max, self.V), dtype=torch.float32, device=dev)
        self.target = torch.zeros((self.B, self.Kt, self.V), dtype=torch.float32, device=dev)
        self.tokens = torch.zeros((self.B, self.K_max), dtype=torch.int32, device=dev)
        self.hist_k = torch.full((self.iterations + 1, self.B), self.K_max, dtype=torch.int32, device=dev)
        self.hist_n = torch.zeros((self.iterations, self.B), dtype=torch.int32, device=dev)
        self.hist_tok = torch.zeros((self.iterations, self.B, self.Kt), dtype=torch.int32, device=dev)
        self.ws = cmsd.workspace(self.B, self.K_max, self.V)
        self._fn = cmsd.lib().cmsd_confidence_verify
        self._gen = wlib().cmsd_gen_decode_rows

    def _ptr(self, t, it=None):
        base = t.data_ptr()
        if it is not None:
            base += it * t.stride(0) * t.element_size()
        return ctypes.c_void_p(base)

    def generate(self, it, stream=None):
        """Device logits of iteration `it` for the rows its window needs."""
        s = cmsd._stream() if stream is None else stream
        rc = self._gen(self._ptr(self.table), self._ptr(self.heights, it), int(it), self.B, self.K_max, self.Kt,
                       self.V, self._ptr(self.hist_k, it), self.seed, self._ptr(self.draft),
                       self._ptr(self.target), self._ptr(self.tokens), s)
        if rc != 0:
            raise cmsd.CmsdError(f"cmsd_gen_decode_rows failed [{rc}]")

    def verify(self, it, stream=None):
        """The fused pass of iteration `it`; k_next lands in hist_k[it + 1]."""
        s = cmsd._stream() if stream is None else stream
        rc = self._fn(self._ptr(self.draft), self._ptr(self.target), self._ptr(self.tokens),
                      self._ptr(self.hist_k, it), self.B, self.K_max, self.V, cmsd.F32, ctypes.byref(self.p),
                      self.seed, int(it), None, None, None, None, None, self._ptr(self.hist_k, it + 1),
                      self._ptr(self.hist_n, it), self._ptr(self.hist_tok, it), None, self._ptr(self.ws),
                      self.ws.numel(), s)
        if rc != cmsd.OK:
            cmsd._check(rc, "cmsd_confidence_verify")

    def step(self, it):
        s = cmsd._stream()
        self.generate(it, s)
        self.verify(it, s)

    def run(self, graph=False):
        """All iterations (replayed from one CUDA graph when `graph`); returns
        per-iteration host arrays k, n_accept, out_tokens."""
        import torch
        if graph:
            g = self.capture()
            g.replay()
        else:
            for it in range(self.iterations):
                self.step(it)
        torch.cuda.current_stream().synchronize()
        return self.history()

    def capture(self, generate=True, verify=True):
        """A CUDA graph of every iteration (generation and / or pass)."""
        import torch
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g):
            s = cmsd._stream()
            for it in range(self.iterations):
                if generate:
                    self.generate(it, s)
                if verify:
                    self.verify(it, s)
        return g

    def history(self):
        return {"k": self.hist_k[:-1].cpu().numpy(), "n_accept": self.hist_n.cpu().numpy(),
                "out_tokens": self.hist_tok.cpu().numpy()}


def pass_bytes(hist, V, elem=4, bonus=False):
    """Logit bytes one loop's passes read: every drafted row pair once, the
    extra verifier row of each sequence (bonus), and the row pair of each
    rejected position again (the residual draw)."""
    k, n = hist["k"].astype(np.int64), hist["n_accept"].astype(np.int64)
    rows = int(k.sum()) * 2 + (k.size if bonus else 0)
    rows += 2 * int((n < k).sum())
    return rows * V * elem


def summarize(hist, bonus=False):
    """Mean drafted and accepted lengths, tokens emitted per iteration (the
    accepted drafts, plus the correction of a rejected position, or with the
    bonus row the verifier's token after a fully accepted window), rollbacks
    and rows verified."""
    k, n = hist["k"].astype(np.int64), hist["n_accept"].astype(np.int64)
    emitted = n + (n < k) + ((n == k) if bonus else 0)
    return {"iterations": int(k.shape[0]), "sequences": int(k.shape[1]),
            "mean_k": float(k.mean()), "mean_accepted": float(n.mean()),
            "tokens_per_iteration": float(emitted.mean()), "rollbacks": int((n < k).sum()),
            "rows": int(k.sum())}
