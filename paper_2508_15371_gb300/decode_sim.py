"""Algorithm 1 as a control loop over synthetic logits (decode-loop simulation).

The paper's drafter and verifier models (Sec. IV.A) are not available, so their
logits are produced on the device by libcmsd_workload.so, bit-identical to the
host recipe in workloads.py (decode_row_host: a drafter row with one spike
whose height drifts per sequence as an AR(1) process, and a noisy verifier).

Each iteration drafts k_row[b] positions of every sequence b, runs the fused
pass of libcmsd.so with that k_row, and feeds the k_next it returns back as the
next iteration's k_row (Sec. III.B(b)): on the device, through two k buffers
used in turn, without a host round trip.  Per-iteration n_accept and out_tokens
are kept on the device and read back once at the end.
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
                                                   ctypes.c_int, vp, ctypes.c_uint64, vp, vp, vp, vp]
                _wlib = L
    return _wlib


class DecodeSim:
    """State of one simulated decode loop: B sequences, window K_max, V logits.

    `p` is a cmsd.Params; `seed` keys both the logit generator and the
    acceptance / residual uniforms of the method.
    """

    def __init__(self, B, K_max, V, iterations, p, seed=4, device="cuda"):
        import torch
        self.B, self.K_max, self.V, self.iterations = int(B), int(K_max), int(V), int(iterations)
        self.p, self.seed = p, int(seed)
        dev = torch.device(device)
        self.table = torch.from_numpy(workloads.normal_table()).to(dev)
        self.heights = torch.from_numpy(workloads.ar1_heights(self.B, self.iterations, self.seed,
                                                              workloads.normal_table())).to(dev)
        self.draft = torch.zeros((self.B, self.K_max, self.V), dtype=torch.float32, device=dev)
        self.target = torch.zeros_like(self.draft)
        self.tokens = torch.zeros((self.B, self.K_max), dtype=torch.int32, device=dev)
        self.k = [torch.full((self.B,), self.K_max, dtype=torch.int32, device=dev),
                  torch.empty((self.B,), dtype=torch.int32, device=dev)]
        self.hist_k = torch.empty((self.iterations, self.B), dtype=torch.int32, device=dev)
        self.hist_n = torch.empty((self.iterations, self.B), dtype=torch.int32, device=dev)
        self.hist_tok = torch.empty((self.iterations, self.B, self.K_max), dtype=torch.int32, device=dev)
        self.ws = cmsd.workspace(self.B, self.K_max, self.V)

    def generate(self, it, k_row):
        """Device logits of iteration `it` for the rows i < k_row[b]."""
        rc = wlib().cmsd_gen_decode_rows(
            cmsd._ptr(self.table), cmsd._ptr(self.heights[it]), int(it), self.B, self.K_max, self.V,
            cmsd._ptr(k_row), self.seed, cmsd._ptr(self.draft), cmsd._ptr(self.target),
            cmsd._ptr(self.tokens), cmsd._stream())
        if rc != 0:
            raise cmsd.CmsdError(f"cmsd_gen_decode_rows failed [{rc}]")

    def step(self, it):
        k_row, k_next = self.k[it % 2], self.k[(it + 1) % 2]
        self.generate(it, k_row)
        o = cmsd.confidence_verify(self.draft, self.target, self.tokens, k_row=k_row, p=self.p,
                                   seed=self.seed, iteration=it, ws=self.ws, signals=False,
                                   out={"k_next": k_next})
        self.hist_k[it].copy_(k_row)
        self.hist_n[it].copy_(o["n_accept"])
        self.hist_tok[it].copy_(o["out_tokens"])

    def run(self):
        """All iterations; returns per-iteration host arrays k, n_accept, out_tokens."""
        import torch
        for it in range(self.iterations):
            self.step(it)
        torch.cuda.current_stream().synchronize()
        return {"k": self.hist_k.cpu().numpy(), "n_accept": self.hist_n.cpu().numpy(),
                "out_tokens": self.hist_tok.cpu().numpy()}


def summarize(hist):
    """Mean drafted and accepted lengths, tokens emitted per iteration (accepted
    drafts plus the correction of a rejected position; no token is added when
    every draft is accepted), rollbacks and rows verified."""
    k, n = hist["k"].astype(np.int64), hist["n_accept"].astype(np.int64)
    emitted = n + (n < k)
    return {"iterations": int(k.shape[0]), "sequences": int(k.shape[1]),
            "mean_k": float(k.mean()), "mean_accepted": float(n.mean()),
            "tokens_per_iteration": float(emitted.mean()), "rollbacks": int((n < k).sum()),
            "rows": int(k.sum())}
