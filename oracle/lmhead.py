"""Oracle for the drafter's LM head followed by the confidence signals --
TEST INFRASTRUCTURE, NOT THE PRODUCT.

The paper puts its confidence estimator on the drafter's output logits: a
light layer over the logits that the drafter's last projection produces
(Sec. I), whose signals are the entropy, logit margin and softmax margin of
Sec. III.B(1).  Those logits are z = h W^T, the drafter's final hidden state
h (length d) times its LM-head weight W (V rows of length d).  This module
restates that composition in float64:

  lm_head_logits       z[r, v] = sum_j h[r, j] W[v, j], bf16 inputs read
                       exactly into float64, one plain matrix product;
  lm_head_confidence   the signals and unified confidence of every row of z,
                       by cmsd_oracle.drafter_signals / unified_confidence
                       (Sec. III.B(1)), which are pinned on their own.

Near-threshold flag: a row whose two largest logits are within `flag_gap`
of each other has its argmax flagged (the CUDA path rounds the dot products
to float32, which can reorder a near-tie); tests skip flagged argmax values
in bit-exact comparisons and count them.

Only tests/, __graft_entry__.smoke() and bench.py's CPU legs may import this.
"""
from __future__ import annotations

import numpy as np

from .cmsd_oracle import Params, bf16_bits_to_f64, drafter_signals, unified_confidence


def lm_head_logits(hidden_bits, weight_bits):
    """Logits z = h W^T of bf16 hidden states [R, d] and LM-head weights [V, d]
    (uint16 bit patterns), in float64."""
    h = bf16_bits_to_f64(hidden_bits)
    w = bf16_bits_to_f64(weight_bits)
    if h.ndim != 2 or w.ndim != 2 or h.shape[1] != w.shape[1]:
        raise ValueError("hidden [R, d] and weight [V, d] must share d")
    return h @ w.T


def lm_head_confidence(hidden_bits, weight_bits, P: Params, rows=None, flag_gap=0.0):
    """Per-row H, margin, psm, argmax, lse and C of the LM head's logits.

    rows: optional iterable of row indices to evaluate (others stay NaN / -1).
    Returns a dict of arrays, plus `logits` (float64, every row) and
    `argmax_flag` (rows whose top-2 gap is <= flag_gap).
    """
    z = lm_head_logits(hidden_bits, weight_bits)
    R, V = z.shape
    out = {k: np.full(R, np.nan) for k in ("H", "margin", "psm", "lse", "conf")}
    out["argmax"] = np.full(R, -1, dtype=np.int64)
    out["argmax_flag"] = np.zeros(R, dtype=bool)
    for r in (range(R) if rows is None else rows):
        s = drafter_signals(z[r])
        for k in ("H", "margin", "psm", "lse"):
            out[k][r] = s[k]
        out["argmax"][r] = s["argmax"]
        out["argmax_flag"][r] = s["margin"] <= flag_gap
        out["conf"][r] = unified_confidence(s["H"], s["margin"], s["psm"], V, P)
    out["logits"] = z
    return out


def signal_error_bound(eps, H, V, lam, beta_sig):
    """How far the signals can move when every logit of a row moves by at most
    eps (first order in eps):
      lse    <= eps
      margin <= 2 eps
      H      <= 2 eps (H + 1)     (d log p_v <= 2 eps, d p_v <= 2 eps p_v)
      psm    <= 4 eps             (|d p1| + |d p2| <= 2 eps (p1 + p2))
      C      <= lam1 dH / log V + lam2 beta_sig dmargin / 4 + lam3 dpsm / (1 - 1/V)
    Returns a dict of bounds."""
    H = np.asarray(H, dtype=np.float64)
    dH = 2.0 * eps * (H + 1.0)
    dm = 2.0 * eps
    dpsm = 4.0 * eps
    dC = lam[0] * dH / np.log(V) + lam[1] * beta_sig * dm / 4.0 + lam[2] * dpsm / (1.0 - 1.0 / V)
    return {"lse": eps, "margin": dm, "H": dH, "psm": dpsm, "conf": dC}
