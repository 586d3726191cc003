"""Oracle for the CM-ASD logits pass -- TEST INFRASTRUCTURE, NOT THE PRODUCT.

A plain, slow, float64 numpy restatement of what one iteration of
confidence-modulated speculative decoding (Sen, Dasgupta, Waghela,
arXiv 2508.15371) computes over vocabulary-wide logits.  It follows the
paper's definitions step by step, in the paper's notation, with no blocking,
fusion or online rescaling.  It shares no code with the CUDA library and
imports nothing from the package; only tests/, __graft_entry__.smoke() and
bench.py's CPU-baseline and reference legs may import it.

Steps and where the paper defines them:

  drafter signals   Sec. III.B(1): entropy C^(ent), normalised by log|V|;
                    logit margin z(1) - z(2) through a sigmoid; softmax
                    margin P(1) - P(2) normalised by (1 - 1/|V|)
  unified score     Sec. III.B(1), "Unified confidence score"
  draft length      Sec. III.B(b): mean confidence over the window, then
                    k = min(k_max, max(k_min, floor(alpha * Cbar * k_max)))
  threshold         Sec. III.B(c): tau_t = tau_base + gamma * (1 - C_t)
  PAPER rule        Sec. III.B(c), "Modified verification rule": top-beta
                    inclusion and log-likelihood gap <= tau_t; halt at the
                    first failure (Sec. III.A(2)); the rejected position is
                    redone by the verifier, i.e. its greedy token.
  SAMPLED rule      speculative sampling of the works cited in Sec. II
                    ([5], [6]), modulated by tau_t: accept with probability
                    min(1, e^tau * p / q), else draw from the normalised
                    residual max(0, p - q) with a two-level exponential race
                    (groups of 32 entries, then entries of the winning group).

Readings where the paper is garbled, silent or self-contradictory (the
reason for each is stated beside it):
  C1  the entropy term enters the ensemble as 1 - H/log|V| (high entropy is
      low confidence, Sec. III.B(b) "low entropy ... Cbar -> 1").
  C2  the garbled "sigma * (beta * (z1 - z2))" is the logistic
      sigma(beta_sig * margin).
  C3  the ensemble is clamped to [0, 1] (the paper requires C_t in [0, 1]).
  C4  Cbar is the mean over the positions present (k_row of them); the
      resulting k drives the next iteration.
  C5  tau_t follows the printed equation (tau_sign = +1); tau_sign = -1
      gives the prose reading tau_base + gamma * C_t.
  C6  the garbled k_j formula is min(k_max, max(k_min, floor(...))).
  C8  argmax ties go to the lowest index; top-beta counts strictly greater
      logits; z(2) is the largest logit at any index other than argmax.
  C9  SAMPLED acceptance probability min(1, e^tau p/q), residual
      max(0, p - q) (tau = 0 gives exact speculative sampling).
  C10 bonus row (optional, Params.bonus): the verifier scores one position
      more than was drafted (Sec. III.A(2): after the accepted prefix the
      verifier's own prediction continues the sequence); when all k drafts
      are accepted, that row gives one more token -- its argmax under the
      PAPER rule, a draw from its softmax under the SAMPLED rule.  Without
      it, no token is added when all k positions are accepted.
  T3  fixed draft length (Params.k_fixed > 0): the "fixed k" variants of the
      ablation in Sec. IV (Table III) replace the adaptive k by a constant.
  C12 uniforms from Philox4x32-10 (oracle/philox.py).
  C13 -inf logits have probability 0 and add nothing to the entropy.
  R1  when the residual is identically zero (possible only with the rank
      gate on in SAMPLED mode), the correction is the target argmax.

Near-threshold flags: a decision that flips under a perturbation of about
1e-6 (relative for probabilities, absolute for the log gap and k) is flagged;
parity tests count flagged decisions and exclude them from bit-exact checks.

Parity unpinned: none of the paper's end-to-end tables (they need WMT /
CNN-DailyMail data and trained models).  Every function here is pinned in
tests/test_oracle_pins.py.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

from . import philox

FLAG_EPS = 1e-6


@dataclass
class Params:
    """Hyper-parameters listed as the inputs of Algorithm 1 (Sec. III.B)."""
    k_min: int = 1
    k_max: int = 8
    lam: tuple = (1.0 / 3.0, 1.0 / 3.0, 1.0 / 3.0)   # (entropy, logit margin, softmax margin)
    beta_sig: float = 1.0       # sigmoid sharpness of the logit margin
    beta_rank: int = 3          # top-beta inclusion; 0 = no rank gate
    alpha: float = 1.0          # aggressiveness, in (0, 1]
    tau_base: float = 0.1
    gamma: float = 1.0
    tau_sign: int = 1           # +1: printed equation; -1: prose reading
    rule: str = "paper"         # "paper" or "sampled"
    k_fixed: int = 0            # > 0: constant draft length (Table III "fixed k")
    bonus: bool = False         # the verifier supplies row k_b after the drafts


# ---------------------------------------------------------------------------
# input conversion
# ---------------------------------------------------------------------------

def bf16_bits_to_f64(bits):
    """bfloat16 bit patterns (uint16) -> float64, exactly."""
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def logits_to_f64(x, dtype):
    if dtype == "bf16":
        return bf16_bits_to_f64(x)
    if dtype == "f32":
        return np.asarray(x, dtype=np.float32).astype(np.float64)
    raise ValueError(f"unknown dtype {dtype!r}")


# ---------------------------------------------------------------------------
# Sec. III.B(1): confidence signals of one drafter row
# ---------------------------------------------------------------------------

def softmax(z):
    z = np.asarray(z, dtype=np.float64)
    m = np.max(z)
    if not np.isfinite(m):
        raise ValueError("row has no finite logit")
    e = np.exp(z - m)
    return e / np.sum(e)


def drafter_signals(z):
    """Entropy, top-2 logit margin and softmax margin of one drafter row.

    Returns a dict with H (natural log), margin = z(1) - z(2), psm = P(1) - P(2),
    argmax (lowest index), lse (log-sum-exp of the row).
    """
    z = np.asarray(z, dtype=np.float64)
    V = z.size
    if V < 2:
        raise ValueError("V must be >= 2")
    i1 = int(np.argmax(z))                     # first index of the maximum
    z1 = z[i1]
    if not np.isfinite(z1):
        raise ValueError("row has no finite logit")
    rest = np.concatenate([z[:i1], z[i1 + 1:]])
    z2 = float(np.max(rest))                   # may equal z1 (duplicated max)
    p = softmax(z)
    pos = p > 0
    H = float(-np.sum(p[pos] * np.log(p[pos])))
    margin = float(z1 - z2)                    # +inf if every other logit is -inf
    s = float(np.sum(np.exp(z - z1)))
    p1 = 1.0 / s
    p2 = math.exp(z2 - z1) / s if np.isfinite(z2) else 0.0
    return {
        "H": H,
        "margin": margin,
        "psm": p1 - p2,
        "argmax": i1,
        "lse": float(z1 + math.log(s)),
    }


def unified_confidence(H, margin, psm, V, P: Params):
    """C_t = lam1 * (1 - H/log|V|) + lam2 * sigma(beta_sig * margin)
             + lam3 * psm / (1 - 1/|V|), clamped to [0, 1] (readings C1-C3)."""
    l1, l2, l3 = P.lam
    c_ent = 1.0 - H / math.log(V)
    x = P.beta_sig * margin
    c_mar = 1.0 / (1.0 + math.exp(-x)) if x > -700 else 0.0
    c_soft = psm / (1.0 - 1.0 / V)
    C = l1 * c_ent + l2 * c_mar + l3 * c_soft
    return min(1.0, max(0.0, C))


# ---------------------------------------------------------------------------
# Sec. III.B(b): draft length
# ---------------------------------------------------------------------------

def next_draft_length(C_window, P: Params):
    """k = min(k_max, max(k_min, floor(alpha * Cbar * k_max))) over the window.

    Returns (k, flagged).  An empty window gives k_min (no signal).
    """
    if P.k_fixed > 0:                          # Table III, fixed k: no adaptation
        return int(P.k_fixed), False
    C_window = [float(c) for c in C_window]
    if not C_window:
        return P.k_min, False
    Cbar = sum(C_window) / len(C_window)
    x = P.alpha * Cbar * P.k_max
    k = min(P.k_max, max(P.k_min, math.floor(x)))
    exact = len(set(C_window)) == 1 and C_window[0] in (0.0, 1.0)
    flagged = (not exact) and abs(x - round(x)) < FLAG_EPS
    return int(k), flagged


# ---------------------------------------------------------------------------
# Sec. III.B(c): confidence-modulated verification
# ---------------------------------------------------------------------------

def tau_t(C, P: Params):
    if P.tau_sign >= 0:
        return P.tau_base + P.gamma * (1.0 - C)
    return P.tau_base + P.gamma * C


def log_softmax(z):
    z = np.asarray(z, dtype=np.float64)
    m = np.max(z)
    return z - (m + math.log(float(np.sum(np.exp(z - m)))))


def rank_gate(zt, tok, beta_rank):
    """Top-beta inclusion: fewer than beta logits strictly above the draft's."""
    if beta_rank <= 0:
        return True
    zt = np.asarray(zt, dtype=np.float64)
    return int(np.sum(zt > zt[tok])) < beta_rank


def accept_paper(zt, tok, tau, beta_rank):
    """PAPER rule. Returns (accepted, flagged)."""
    logp = log_softmax(zt)
    gap = float(np.max(logp) - logp[tok])
    ok_rank = rank_gate(zt, tok, beta_rank)
    acc = ok_rank and gap <= tau
    flagged = ok_rank and abs(gap - tau) < FLAG_EPS
    return acc, flagged


def accept_sampled(zt, zd, tok, tau, u, beta_rank):
    """SAMPLED rule: accept iff u * q(tok) < e^tau * p(tok) (and the optional
    rank gate). Returns (accepted, flagged, p, q)."""
    p = float(softmax(zt)[tok])
    q = float(softmax(zd)[tok])
    lhs = u * q
    rhs = math.exp(tau) * p
    ok_rank = rank_gate(zt, tok, beta_rank)
    acc = ok_rank and lhs < rhs
    flagged = ok_rank and abs(lhs - rhs) < FLAG_EPS * max(lhs, rhs)
    return acc, flagged, p, q


def _race(keys_E, rates, eps=FLAG_EPS, r_lo=None, r_hi=None):
    """Exponential race: winner = argmin over rates > 0 of E / rate (lowest index
    on ties).  Returns (winner or -1, flagged); flagged when the winner could
    change under the given interval [r_lo, r_hi] of each rate and relative eps
    on each E."""
    E = np.asarray(keys_E, dtype=np.float64)
    r = np.asarray(rates, dtype=np.float64)
    cand = r > 0
    if not np.any(cand):
        return -1, False
    with np.errstate(divide="ignore", invalid="ignore"):
        key = np.where(cand, E / np.where(cand, r, 1.0), np.inf)
    w = int(np.argmin(key))
    if r_lo is None:
        return w, False
    with np.errstate(divide="ignore", invalid="ignore"):
        key_lo = np.where(r_hi > 0, E * (1 - eps) / np.where(r_hi > 0, r_hi, 1.0), np.inf)
    key_hi_w = E[w] * (1 + eps) / r_lo[w] if r_lo[w] > 0 else np.inf
    key_lo[w] = np.inf
    return w, bool(key_hi_w >= np.min(key_lo))


def two_level_race(r, r_lo, r_hi, seed, b, n, iteration):
    """Draw from norm(r) (r >= 0, not all 0) with a two-level exponential race.

    The vocabulary is cut into groups of philox.GROUP = 32 consecutive
    entries with mass R_g = sum of r_v over the group.  Level 1: group g gets
    E_g = -log(1 - U_g) and the winning group is argmin E_g / R_g (law
    R_g / R).  Level 2: inside the winning group, entry v gets
    E_v = -log(1 - U_v) and the token is argmin E_v / r_v (law r_v / R_g).
    Together the token has law r_v / R.  Ties go to the lowest index.  The
    uniforms are those of position n of sequence b (oracle/philox.py).
    Returns (token, flagged); flagged when either level's winner could change
    with each rate anywhere in [r_lo, r_hi] and the exponentials perturbed by
    a relative FLAG_EPS.
    """
    eps = FLAG_EPS
    V = r.size
    G = philox.GROUP
    ng = (V + G - 1) // G
    pad = ng * G - V
    R = np.pad(r, (0, pad)).reshape(ng, G).sum(axis=1)
    R_hi = np.pad(r_hi, (0, pad)).reshape(ng, G).sum(axis=1)
    R_lo = np.pad(r_lo, (0, pad)).reshape(ng, G).sum(axis=1)
    Ug = philox.group_uniforms(seed, b, n, iteration, ng)
    g, f1 = _race(-np.log1p(-Ug), R, eps, R_lo, R_hi)
    v0, v1 = g * G, min(V, (g + 1) * G)
    Uv = philox.residual_uniforms(seed, b, n, iteration, V)[v0:v1]
    k, f2 = _race(-np.log1p(-Uv), r[v0:v1], eps, r_lo[v0:v1], r_hi[v0:v1])
    return v0 + k, bool(f1 or f2)


def residual_token(zt, zd, seed, b, n, iteration):
    """Draw from norm(max(0, p - q)) at the rejected position n (reading C9).

    r_v = max(0, p_v - q_v) with p the verifier's and q the drafter's softmax;
    the draw is the two-level race above.  If r is identically 0 the
    correction is the verifier's argmax (reading R1).  Returns (token,
    flagged); the rate bounds perturb p and q by a relative FLAG_EPS.
    """
    p = softmax(zt)
    q = softmax(zd)
    r = np.maximum(0.0, p - q)
    if not np.any(r > 0):
        return int(np.argmax(np.asarray(zt, dtype=np.float64))), False   # reading R1
    eps = FLAG_EPS
    r_hi = np.maximum(0.0, p * (1 + eps) - q * (1 - eps))
    r_lo = np.maximum(0.0, p * (1 - eps) - q * (1 + eps))
    return two_level_race(r, r_lo, r_hi, seed, b, n, iteration)


def bonus_token(zt, rule, seed, b, n, iteration):
    """The token of the verifier's extra row n = k_b when all drafts were
    accepted (reading C10): its argmax (lowest index) under the PAPER rule,
    a draw from its softmax p under the SAMPLED rule (the two-level race with
    r = p, using the uniforms of position n, which no residual draw of this
    iteration uses since a residual position is always below k_b).
    Returns (token, flagged)."""
    zt = np.asarray(zt, dtype=np.float64)
    if rule == "paper":
        return int(np.argmax(zt)), False
    p = softmax(zt)
    eps = FLAG_EPS
    return two_level_race(p, p * (1 - eps), p * (1 + eps), seed, b, n, iteration)


# ---------------------------------------------------------------------------
# one iteration over a batch
# ---------------------------------------------------------------------------

@dataclass
class Result:
    H: np.ndarray
    margin: np.ndarray
    psm: np.ndarray
    argmax: np.ndarray
    conf: np.ndarray
    lse: np.ndarray
    k_next: np.ndarray
    k_flag: np.ndarray
    accept: np.ndarray = None
    acc_flag: np.ndarray = None
    n_accept: np.ndarray = None
    n_flag: np.ndarray = None
    out_tokens: np.ndarray = None
    tok_flag: np.ndarray = None
    target_argmax: np.ndarray = None
    extra: dict = field(default_factory=dict)


def _k_rows(B, K, k_row):
    if k_row is None:
        return np.full(B, K, dtype=np.int64)
    k = np.asarray(k_row, dtype=np.int64)
    if k.shape != (B,) or np.any(k < 0) or np.any(k > K):
        raise ValueError("k_row must have shape (B,) with 0 <= k_row <= K")
    return k


def confidence(draft, P: Params, k_row=None, rows=None):
    """Confidence pass over drafter logits draft[B, K, V] (float64).

    rows: optional iterable of (b, i) to evaluate (others are left NaN / -1).
    k_next is computed only for sequences whose rows were all evaluated.
    """
    draft = np.asarray(draft, dtype=np.float64)
    B, K, V = draft.shape
    kb = _k_rows(B, K, k_row)
    H = np.full((B, K), np.nan)
    margin = np.full((B, K), np.nan)
    psm = np.full((B, K), np.nan)
    lse = np.full((B, K), np.nan)
    conf = np.full((B, K), np.nan)
    argmax = np.full((B, K), -1, dtype=np.int64)
    want = set(rows) if rows is not None else None
    for b in range(B):
        for i in range(int(kb[b])):
            if want is not None and (b, i) not in want:
                continue
            sig = drafter_signals(draft[b, i])
            H[b, i] = sig["H"]
            margin[b, i] = sig["margin"]
            psm[b, i] = sig["psm"]
            argmax[b, i] = sig["argmax"]
            lse[b, i] = sig["lse"]
            conf[b, i] = unified_confidence(sig["H"], sig["margin"], sig["psm"], V, P)
    k_next = np.full(B, -1, dtype=np.int64)
    k_flag = np.zeros(B, dtype=bool)
    for b in range(B):
        window = conf[b, : int(kb[b])]
        if np.all(np.isfinite(window)):
            k_next[b], k_flag[b] = next_draft_length(window, P)
    return Result(H=H, margin=margin, psm=psm, argmax=argmax, conf=conf, lse=lse,
                  k_next=k_next, k_flag=k_flag)


def verify_sequence(draft_b, target_b, tokens_b, conf_b, k_b, P: Params, seed, b, iteration):
    """Verification of one sequence: per-position accept, first failure, correction.

    With P.bonus the verifier rows target_b hold one more row than drafted
    (row k_b is the bonus row, reading C10) and out_tokens has K + 1 entries.
    Returns dict with accept[k_b], acc_flag[k_b], n_accept, n_flag,
    out_tokens[K (+1)], tok_flag, target_argmax[k_b].
    """
    K = len(tokens_b)
    acc = np.zeros(k_b, dtype=bool)
    aflag = np.zeros(k_b, dtype=bool)
    targmax = np.full(k_b, -1, dtype=np.int64)
    for i in range(k_b):
        zt = target_b[i]
        tok = int(tokens_b[i])
        tau = tau_t(float(conf_b[i]), P)
        targmax[i] = int(np.argmax(zt))
        if P.rule == "paper":
            acc[i], aflag[i] = accept_paper(zt, tok, tau, P.beta_rank)
        elif P.rule == "sampled":
            u = philox.accept_uniform(seed, b, i, iteration)
            acc[i], aflag[i], _, _ = accept_sampled(zt, draft_b[i], tok, tau, u, P.beta_rank)
        else:
            raise ValueError(P.rule)
    # Sec. III.A(2) / III.B(c): halt at the first failure
    n = k_b
    for i in range(k_b):
        if not acc[i]:
            n = i
            break
    n_flag = bool(np.any(aflag[: min(n + 1, k_b)]))
    out = np.full(K + 1 if P.bonus else K, -1, dtype=np.int64)
    out[:n] = np.asarray(tokens_b[:n], dtype=np.int64)
    tok_flag = n_flag
    if n < k_b:
        if P.rule == "paper":
            out[n] = targmax[n]
        else:
            out[n], rflag = residual_token(target_b[n], draft_b[n], seed, b, n, iteration)
            tok_flag = tok_flag or rflag
    elif P.bonus:                               # every draft accepted: the verifier's own token
        out[k_b], rflag = bonus_token(target_b[k_b], P.rule, seed, b, k_b, iteration)
        tok_flag = tok_flag or rflag
    return {"accept": acc, "acc_flag": aflag, "n_accept": n, "n_flag": n_flag,
            "out_tokens": out, "tok_flag": tok_flag, "target_argmax": targmax}


def confidence_verify(draft, target, tokens, P: Params, seed=0, iteration=0,
                      k_row=None, seqs=None):
    """Full iteration: confidence signals, k_next, verification, correction.

    draft: float64 [B, K, V]; target: float64 [B, K, V], or [B, K + 1, V]
    with P.bonus; tokens: int [B, K].
    seqs: optional list of sequence indices to evaluate (others left empty).
    """
    draft = np.asarray(draft, dtype=np.float64)
    target = np.asarray(target, dtype=np.float64)
    tokens = np.asarray(tokens)
    B, K, V = draft.shape
    kb = _k_rows(B, K, k_row)
    seq_list = list(range(B)) if seqs is None else list(seqs)
    rows = [(b, i) for b in seq_list for i in range(int(kb[b]))]
    res = confidence(draft, P, k_row=k_row, rows=rows)
    res.accept = np.zeros((B, K), dtype=bool)
    res.acc_flag = np.zeros((B, K), dtype=bool)
    res.n_accept = np.full(B, -1, dtype=np.int64)
    res.n_flag = np.zeros(B, dtype=bool)
    res.out_tokens = np.full((B, K + 1 if P.bonus else K), -1, dtype=np.int64)
    res.tok_flag = np.zeros(B, dtype=bool)
    res.target_argmax = np.full((B, K), -1, dtype=np.int64)
    for b in seq_list:
        k_b = int(kb[b])
        v = verify_sequence(draft[b], target[b], tokens[b], res.conf[b], k_b, P, seed, b, iteration)
        res.accept[b, :k_b] = v["accept"]
        res.acc_flag[b, :k_b] = v["acc_flag"]
        res.n_accept[b] = v["n_accept"]
        res.n_flag[b] = v["n_flag"]
        res.out_tokens[b] = v["out_tokens"]
        res.tok_flag[b] = v["tok_flag"]
        res.target_argmax[b, :k_b] = v["target_argmax"]
    return res


def verify(draft, target, tokens, conf, P: Params, seed=0, iteration=0, k_row=None):
    """Verification only, given the confidence scores of every present position."""
    draft = np.asarray(draft, dtype=np.float64)
    target = np.asarray(target, dtype=np.float64)
    B, K, V = draft.shape
    kb = _k_rows(B, K, k_row)
    out = {"accept": np.zeros((B, K), dtype=bool), "acc_flag": np.zeros((B, K), dtype=bool),
           "n_accept": np.zeros(B, dtype=np.int64), "n_flag": np.zeros(B, dtype=bool),
           "out_tokens": np.full((B, K + 1 if P.bonus else K), -1, dtype=np.int64),
           "tok_flag": np.zeros(B, dtype=bool)}
    for b in range(B):
        k_b = int(kb[b])
        v = verify_sequence(draft[b], target[b], tokens[b], conf[b], k_b, P, seed, b, iteration)
        out["accept"][b, :k_b] = v["accept"]
        out["acc_flag"][b, :k_b] = v["acc_flag"]
        out["n_accept"][b] = v["n_accept"]
        out["n_flag"][b] = v["n_flag"]
        out["out_tokens"][b] = v["out_tokens"]
        out["tok_flag"][b] = v["tok_flag"]
    return out


# ---------------------------------------------------------------------------
# Algorithm 1 as a control loop over generated logits (decode simulation)
# ---------------------------------------------------------------------------

def decode_sim_sequence(gen_rows, b, iterations, K_max, P: Params, seed):
    """Replay the draft-length / acceptance trajectory of sequence b.

    gen_rows(it, b, k) -> (draft[k, V], target[k, V], tokens[k]) supplies the
    drafted positions present at iteration it (float arrays; with P.bonus the
    target has k + 1 rows, the last being the bonus row).  The first
    iteration drafts K_max positions; each later one drafts the k chosen from
    the previous iteration's confidence (reading C4).  Returns a list of dicts
    (k, n_accept, k_next, out_tokens, flagged) per iteration; `flagged` marks
    the first iteration whose k_next or n_accept sits at a decision threshold
    (later iterations then depend on a float-order tie and are not compared).
    """
    k = K_max
    traj = []
    for it in range(iterations):
        d, t, tok = gen_rows(it, b, k)
        d = np.asarray(d, dtype=np.float64)
        t = np.asarray(t, dtype=np.float64)
        V = d.shape[-1]
        conf = np.empty(k)
        for i in range(k):
            s = drafter_signals(d[i])
            conf[i] = unified_confidence(s["H"], s["margin"], s["psm"], V, P)
        k_next, kflag = next_draft_length(conf, P)
        toks = np.full(K_max, -1, dtype=np.int64)
        toks[:k] = tok
        dd = np.zeros((K_max, V))
        tt = np.zeros((K_max + 1 if P.bonus else K_max, V))
        dd[:k] = d
        tt[:t.shape[0]] = t
        v = verify_sequence(dd, tt, toks, np.concatenate([conf, np.zeros(K_max - k)]), k, P,
                            seed, b, it)
        traj.append({"k": k, "n_accept": v["n_accept"], "k_next": k_next,
                     "out_tokens": v["out_tokens"], "flagged": bool(kflag or v["n_flag"] or v["tok_flag"])})
        k = k_next
    return traj
