"""Thin Python binding of libcmsd.so (ctypes).

Argument marshalling only: torch supplies device memory and the current
stream; every step of the logits pass runs in the library's CUDA kernels.
There is no CPU fallback -- if libcmsd.so is missing or fails to load, every
call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libcmsd.so")

F32, BF16 = 0, 1
RULE_PAPER, RULE_SAMPLED = 0, 1
OK, EINVAL, EDTYPE, ECUDA, ENOWS, EALIGN, ESCRATCH = 0, -1, -2, -3, -4, -5, -6

_c_int, _c_u32, _c_u64, _c_sz, _vp = ctypes.c_int, ctypes.c_uint32, ctypes.c_uint64, ctypes.c_size_t, ctypes.c_void_p


class Params(ctypes.Structure):
    """cmsd_params (include/cmsd.h)."""
    _fields_ = [
        ("k_min", ctypes.c_int32), ("k_max", ctypes.c_int32),
        ("lam", ctypes.c_float * 3),
        ("beta_sig", ctypes.c_float),
        ("beta_rank", ctypes.c_int32),
        ("alpha", ctypes.c_float),
        ("tau_base", ctypes.c_float),
        ("gamma", ctypes.c_float),
        ("tau_sign", ctypes.c_int32),
        ("rule", ctypes.c_int32),
        ("k_fixed", ctypes.c_int32),
        ("bonus", ctypes.c_int32),
    ]

    def as_dict(self):
        return dict(k_min=self.k_min, k_max=self.k_max, lam=tuple(float(x) for x in self.lam),
                    beta_sig=float(self.beta_sig), beta_rank=self.beta_rank, alpha=float(self.alpha),
                    tau_base=float(self.tau_base), gamma=float(self.gamma), tau_sign=self.tau_sign,
                    rule="sampled" if self.rule == RULE_SAMPLED else "paper", k_fixed=self.k_fixed,
                    bonus=bool(self.bonus))


class CmsdError(RuntimeError):
    pass


_lib = None
_lib_lock = threading.Lock()

_SIGS = {
    "cmsd_params_default": (None, [_vp, _c_int, _c_int]),
    "cmsd_params_preset": (_c_int, [_vp, _c_int, _c_int, _c_int]),
    "cmsd_workspace_bytes": (_c_sz, [_c_int, _c_int, _c_int]),
    "cmsd_workspace_init": (_c_int, [_vp, _c_sz, _vp]),
    "cmsd_workspace_errors": (_c_int, [_vp, _c_sz, _vp, ctypes.POINTER(ctypes.c_uint32)]),
    "cmsd_test_record_wait_timeout": (_c_int, [_vp, _vp, _c_int, _c_int, _c_int, _c_int, _vp, _vp, _c_sz, _vp]),
    "cmsd_confidence": (_c_int, [_vp, _c_int, _c_int, _c_int, _c_int, _vp, _vp,
                                 _vp, _vp, _vp, _vp, _vp, _vp, _vp, _c_sz, _vp]),
    "cmsd_verify": (_c_int, [_vp, _vp, _vp, _vp, _c_int, _c_int, _c_int, _c_int, _vp,
                             _vp, _vp, _c_u64, _c_u32, _vp, _vp, _vp, _vp, _c_sz, _vp]),
    "cmsd_confidence_verify": (_c_int, [_vp, _vp, _vp, _vp, _c_int, _c_int, _c_int, _c_int, _vp,
                                        _c_u64, _c_u32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                        _vp, _c_sz, _vp]),
    "cmsd_confidence_verify_static": (_c_int, [_vp, _vp, _vp, _vp, _c_int, _c_int, _c_int, _c_int, _vp,
                                               _c_u64, _c_u32, _vp, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                               _vp, _vp]),
    "cmsd_lmhead_workspace_bytes": (_c_sz, [_c_int, _c_int, _c_int]),
    "cmsd_lmhead_confidence": (_c_int, [_vp, _vp, _c_int, _c_int, _c_int, _vp, _vp, _vp, _vp, _vp, _vp,
                                        _vp, _vp, _c_sz, _vp]),
    "cmsd_philox_u32": (_c_u32, [_c_u64, _c_u32, _c_u32, _c_u32, _c_u32, _c_int]),
    "cmsd_philox_fill": (_c_int, [_c_u64, _c_u32, _c_u32, _c_u32, _c_u32, _vp, _c_sz, _vp]),
    "cmsd_profile_start": (_c_int, [_c_int]),
    "cmsd_profile_stop": (_c_int, [_vp, _vp, _c_int, ctypes.POINTER(ctypes.c_int)]),
    "cmsd_launch_info": (_c_int, [_c_int, ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_int)]),
    "cmsd_strerror": (ctypes.c_char_p, [_c_int]),
    "cmsd_last_cuda_error": (_c_int, []),
}


def lib():
    """The loaded libcmsd.so (raises if it is missing)."""
    global _lib
    if _lib is None:
        with _lib_lock:
            if _lib is None:
                if not os.path.exists(LIB_PATH):
                    raise CmsdError(f"{LIB_PATH} is missing: build it with "
                                    "`python -c 'import __graft_entry__ as g; g.build()'`")
                L = ctypes.CDLL(LIB_PATH)
                for name, (res, args) in _SIGS.items():
                    fn = getattr(L, name)
                    fn.restype = res
                    fn.argtypes = args
                _lib = L
    return _lib


def _check(rc, what):
    if rc != OK:
        msg = lib().cmsd_strerror(rc).decode()
        if rc == ECUDA:
            msg += f" (cudaError {lib().cmsd_last_cuda_error()})"
        raise CmsdError(f"{what}: {msg} [{rc}]")


PRESETS = {"full": 0, "fixed_k": 1, "fixed_tau": 2, "fixed_k_tau": 3, "entropy_only": 4,
           "margin_only": 5, "softmax_only": 6}


def params(K, rule="paper", preset="full", **kw):
    """cmsd_params for window K, rule ('paper' or 'sampled') and ablation
    preset (PRESETS: the variants of Table III), then overrides.

    Keyword names: k_min, k_max, lam (3-tuple), beta_sig, beta_rank, alpha,
    tau_base, gamma, tau_sign, k_fixed, bonus.
    """
    r = RULE_SAMPLED if rule in ("sampled", RULE_SAMPLED) else RULE_PAPER
    p = Params()
    _check(lib().cmsd_params_preset(ctypes.byref(p), int(K), r, PRESETS[preset]), "cmsd_params_preset")
    for k, v in kw.items():
        if k == "lam":
            for j in range(3):
                p.lam[j] = float(v[j])
        elif k == "rule":
            p.rule = RULE_SAMPLED if v in ("sampled", RULE_SAMPLED) else RULE_PAPER
        elif k == "bonus":
            p.bonus = 1 if v else 0
        else:
            setattr(p, k, v)
    return p


def _torch():
    import torch
    return torch


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dtype_code(t):
    torch = _torch()
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise CmsdError(f"logits must be float32 or bfloat16, got {t.dtype}")


def _check_target(draft, target, p):
    B, K, V = draft.shape
    want = (B, K + 1, V) if p.bonus else (B, K, V)
    if draft.dtype != target.dtype or tuple(target.shape) != want:
        raise CmsdError(f"target logits must be {want} of the drafter's dtype, got {tuple(target.shape)}")


def _stream():
    torch = _torch()
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _need_cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise CmsdError("all tensors must be CUDA tensors (the library has no CPU path)")
        if t is not None and not t.is_contiguous():
            raise CmsdError("tensors must be contiguous")


_ws_cache = {}
_ws_lock = threading.Lock()


def workspace(B, K, V, device=None):
    """A zero-initialised workspace for (B, K, V), cached per device."""
    torch = _torch()
    dev = torch.device("cuda", torch.cuda.current_device() if device is None else device)
    key = (dev.index, B, K, V)
    with _ws_lock:
        ws = _ws_cache.get(key)
        if ws is None:
            n = int(lib().cmsd_workspace_bytes(B, K, V))
            if n == 0:
                raise CmsdError("cmsd_workspace_bytes failed")
            ws = torch.empty(n, dtype=torch.uint8, device=dev)
            _check(lib().cmsd_workspace_init(_ptr(ws), n, _stream()), "cmsd_workspace_init")
            _ws_cache[key] = ws
    return ws


def workspace_errors(ws):
    f = ctypes.c_uint32(0)
    _check(lib().cmsd_workspace_errors(_ptr(ws), ws.numel(), _stream(), ctypes.byref(f)),
           "cmsd_workspace_errors")
    return int(f.value)


def _out(out, name, shape, dtype, device, want=True):
    torch = _torch()
    if out is not None and name in out:
        return out[name]
    if not want:
        return None
    return torch.empty(shape, dtype=dtype, device=device)


def confidence(draft, k_row=None, p=None, out=None, ws=None):
    """Confidence pass; returns dict H, margin, argmax, conf, lse, k_next (torch tensors)."""
    torch = _torch()
    _need_cuda(draft, k_row)
    B, K, V = draft.shape
    p = p if p is not None else params(K)
    dev = draft.device
    o = {n: _out(out, n, (B, K), torch.float32, dev) for n in ("H", "margin", "conf", "lse")}
    o["argmax"] = _out(out, "argmax", (B, K), torch.int32, dev)
    o["k_next"] = _out(out, "k_next", (B,), torch.int32, dev)
    ws = ws if ws is not None else workspace(B, K, V)
    rc = lib().cmsd_confidence(_ptr(draft), B, K, V, _dtype_code(draft), _ptr(k_row), ctypes.byref(p),
                               _ptr(o["H"]), _ptr(o["margin"]), _ptr(o["argmax"]), _ptr(o["conf"]),
                               _ptr(o["lse"]), _ptr(o["k_next"]), _ptr(ws), ws.numel(), _stream())
    _check(rc, "cmsd_confidence")
    return o


def lmhead_workspace(R, d, V):
    """A workspace for cmsd_lmhead_confidence(R, d, V) on the current device."""
    torch = _torch()
    n = int(lib().cmsd_lmhead_workspace_bytes(R, d, V))
    if n == 0:
        raise CmsdError("cmsd_lmhead_workspace_bytes failed")
    return torch.empty(n, dtype=torch.uint8, device="cuda")


def lmhead_confidence(hidden, weight, p=None, logits=False, out=None, ws=None):
    """The drafter's LM head fused with the confidence signals.

    hidden: bf16 [R, d] (torch.bfloat16 or int16/uint16 bits), weight: bf16
    [V, d].  Returns dict H, margin, argmax, conf, lse ([R]) and, with
    logits=True, the fp32 logits [R, V]."""
    torch = _torch()
    _need_cuda(hidden, weight)
    if hidden.element_size() != 2 or weight.element_size() != 2:
        raise CmsdError("hidden and weight must hold 16-bit (bf16) values")
    R, d = hidden.shape
    V, d2 = weight.shape
    if d2 != d:
        raise CmsdError("hidden [R, d] and weight [V, d] must share d")
    p = p if p is not None else params(1)
    dev = hidden.device
    o = {n: _out(out, n, (R,), torch.float32, dev) for n in ("H", "margin", "conf", "lse")}
    o["argmax"] = _out(out, "argmax", (R,), torch.int32, dev)
    if logits:
        o["logits"] = _out(out, "logits", (R, V), torch.float32, dev)
    ws = ws if ws is not None else lmhead_workspace(R, d, V)
    rc = lib().cmsd_lmhead_confidence(_ptr(hidden), _ptr(weight), R, d, V, ctypes.byref(p), _ptr(o["H"]),
                                      _ptr(o["margin"]), _ptr(o["argmax"]), _ptr(o["conf"]), _ptr(o["lse"]),
                                      _ptr(o.get("logits")), _ptr(ws), ws.numel(), _stream())
    _check(rc, "cmsd_lmhead_confidence")
    return o


def verify(draft, target, tokens, conf, draft_lse=None, k_row=None, p=None, seed=0, iteration=0,
           out=None, ws=None):
    """Verification given conf (and draft_lse for the sampled rule); returns n_accept, out_tokens, accept."""
    torch = _torch()
    _need_cuda(draft, target, tokens, conf, draft_lse, k_row)
    B, K, V = draft.shape
    p = p if p is not None else params(K)
    _check_target(draft, target, p)
    dev = draft.device
    o = {"n_accept": _out(out, "n_accept", (B,), torch.int32, dev),
         "out_tokens": _out(out, "out_tokens", (B, K + 1 if p.bonus else K), torch.int32, dev),
         "accept": _out(out, "accept", (B, K), torch.uint8, dev)}
    ws = ws if ws is not None else workspace(B, K, V)
    rc = lib().cmsd_verify(_ptr(draft), _ptr(target), _ptr(tokens), _ptr(k_row), B, K, V,
                           _dtype_code(draft), ctypes.byref(p), _ptr(conf), _ptr(draft_lse),
                           int(seed), int(iteration), _ptr(o["n_accept"]), _ptr(o["out_tokens"]),
                           _ptr(o["accept"]), _ptr(ws), ws.numel(), _stream())
    _check(rc, "cmsd_verify")
    return o


def confidence_verify(draft, target, tokens, k_row=None, p=None, seed=0, iteration=0, out=None,
                      ws=None, signals=True):
    """The fused pass.  Returns n_accept, out_tokens, k_next, accept and (signals=True)
    H, margin, argmax, conf, lse."""
    torch = _torch()
    _need_cuda(draft, target, tokens, k_row)
    B, K, V = draft.shape
    p = p if p is not None else params(K)
    _check_target(draft, target, p)
    dev = draft.device
    o = {}
    for n in ("H", "margin", "conf", "lse"):
        o[n] = _out(out, n, (B, K), torch.float32, dev, signals)
    o["argmax"] = _out(out, "argmax", (B, K), torch.int32, dev, signals)
    o["k_next"] = _out(out, "k_next", (B,), torch.int32, dev)
    o["n_accept"] = _out(out, "n_accept", (B,), torch.int32, dev)
    o["out_tokens"] = _out(out, "out_tokens", (B, K + 1 if p.bonus else K), torch.int32, dev)
    o["accept"] = _out(out, "accept", (B, K), torch.uint8, dev, signals)
    ws = ws if ws is not None else workspace(B, K, V)
    rc = lib().cmsd_confidence_verify(
        _ptr(draft), _ptr(target), _ptr(tokens), _ptr(k_row), B, K, V, _dtype_code(draft),
        ctypes.byref(p), int(seed), int(iteration), _ptr(o["H"]), _ptr(o["margin"]), _ptr(o["argmax"]),
        _ptr(o["conf"]), _ptr(o["lse"]), _ptr(o["k_next"]), _ptr(o["n_accept"]), _ptr(o["out_tokens"]),
        _ptr(o["accept"]), _ptr(ws), ws.numel(), _stream())
    _check(rc, "cmsd_confidence_verify")
    return o


def confidence_verify_static(draft, target, tokens, k_row=None, p=None, seed=0, iteration=0, out=None,
                             signals=True):
    """The fused pass through cmsd_confidence_verify_static: the library's own
    fixed device scratch instead of a workspace (nothing is allocated for it).
    Output tensors are allocated here unless passed in `out`; a caller that may
    not allocate passes them all.  Calls on one device must not overlap."""
    torch = _torch()
    _need_cuda(draft, target, tokens, k_row)
    B, K, V = draft.shape
    p = p if p is not None else params(K)
    _check_target(draft, target, p)
    dev = draft.device
    o = {}
    for n in ("H", "margin", "conf", "lse"):
        o[n] = _out(out, n, (B, K), torch.float32, dev, signals)
    o["argmax"] = _out(out, "argmax", (B, K), torch.int32, dev, signals)
    o["k_next"] = _out(out, "k_next", (B,), torch.int32, dev)
    o["n_accept"] = _out(out, "n_accept", (B,), torch.int32, dev)
    o["out_tokens"] = _out(out, "out_tokens", (B, K + 1 if p.bonus else K), torch.int32, dev)
    o["accept"] = _out(out, "accept", (B, K), torch.uint8, dev, signals)
    rc = lib().cmsd_confidence_verify_static(
        _ptr(draft), _ptr(target), _ptr(tokens), _ptr(k_row), B, K, V, _dtype_code(draft),
        ctypes.byref(p), int(seed), int(iteration), _ptr(o["H"]), _ptr(o["margin"]), _ptr(o["argmax"]),
        _ptr(o["conf"]), _ptr(o["lse"]), _ptr(o["k_next"]), _ptr(o["n_accept"]), _ptr(o["out_tokens"]),
        _ptr(o["accept"]), _stream())
    _check(rc, "cmsd_confidence_verify_static")
    return o


def philox_u32(seed, c0, c1, c2, c3, word):
    return int(lib().cmsd_philox_u32(int(seed), c0, c1, c2, c3, int(word)))


def philox_fill(seed, c0, c1, c2, c3, n, device="cuda"):
    torch = _torch()
    out = torch.empty(n, dtype=torch.int32, device=device)
    _check(lib().cmsd_philox_fill(int(seed), c0, c1, c2, c3, _ptr(out), n, _stream()), "cmsd_philox_fill")
    return out


def profile_start(max_calls):
    _check(lib().cmsd_profile_start(int(max_calls)), "cmsd_profile_start")


def profile_stop(max_calls):
    """Per-call (streaming-kernel ms, resample-kernel ms) recorded since profile_start
    (the second is 0 for calls without a resample kernel)."""
    a = (ctypes.c_float * max(1, max_calls))()
    b = (ctypes.c_float * max(1, max_calls))()
    n = ctypes.c_int(0)
    _check(lib().cmsd_profile_stop(a, b, int(max_calls), ctypes.byref(n)), "cmsd_profile_stop")
    return [float(a[j]) for j in range(n.value)], [float(b[j]) for j in range(n.value)]


def launch_info(dtype=BF16):
    w, s = ctypes.c_int(0), ctypes.c_int(0)
    _check(lib().cmsd_launch_info(int(dtype), ctypes.byref(w), ctypes.byref(s)), "cmsd_launch_info")
    return w.value, s.value


def to_device_logits(arr, dtype, device="cuda"):
    """numpy logits (float32, or uint16 bfloat16 bit patterns) -> CUDA tensor."""
    torch = _torch()
    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(arr).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(arr, dtype=np.float32))
    return t.to(device)


class FusedCall:
    """cmsd_confidence_verify with its arguments marshalled once.

    For tight loops (benchmarks, decode loops): calling the object re-issues
    the same C call on the current stream, optionally with another iteration
    number.  Holds references to every tensor it points at.
    """

    def __init__(self, draft, target, tokens, p, seed=0, iteration=0, k_row=None, out=None, ws=None,
                 signals=False):
        torch = _torch()
        _need_cuda(draft, target, tokens, k_row)
        B, K, V = draft.shape
        dev = draft.device
        o = dict(out or {})
        for n in ("H", "margin", "conf", "lse"):
            o.setdefault(n, torch.empty((B, K), dtype=torch.float32, device=dev) if signals else None)
        o.setdefault("argmax", torch.empty((B, K), dtype=torch.int32, device=dev) if signals else None)
        o.setdefault("accept", torch.empty((B, K), dtype=torch.uint8, device=dev) if signals else None)
        o.setdefault("k_next", torch.empty((B,), dtype=torch.int32, device=dev))
        o.setdefault("n_accept", torch.empty((B,), dtype=torch.int32, device=dev))
        o.setdefault("out_tokens", torch.empty((B, K + 1 if p.bonus else K), dtype=torch.int32, device=dev))
        self.out = o
        self.ws = ws if ws is not None else workspace(B, K, V)
        self._keep = (draft, target, tokens, k_row, p)
        self.p = p
        self.seed = int(seed)
        self.iteration = int(iteration)
        self._fn = lib().cmsd_confidence_verify
        self._head = (_ptr(draft), _ptr(target), _ptr(tokens), _ptr(k_row), B, K, V, _dtype_code(draft),
                      ctypes.byref(p))
        self._tail = (_ptr(o["H"]), _ptr(o["margin"]), _ptr(o["argmax"]), _ptr(o["conf"]), _ptr(o["lse"]),
                      _ptr(o["k_next"]), _ptr(o["n_accept"]), _ptr(o["out_tokens"]), _ptr(o["accept"]),
                      _ptr(self.ws), self.ws.numel())

    def __call__(self, iteration=None, stream=None):
        it = self.iteration if iteration is None else int(iteration)
        s = _stream() if stream is None else ctypes.c_void_p(stream)
        rc = self._fn(*self._head, self.seed, it, *self._tail, s)
        if rc != OK:
            _check(rc, "cmsd_confidence_verify")
        return self.out
