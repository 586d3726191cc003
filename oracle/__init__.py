"""CPU oracle for the CM-ASD logits pass -- test infrastructure only.

Only tests/, __graft_entry__.smoke() and bench.py (its CPU-baseline and
reference legs) may import this package.  It imports nothing from the CUDA
library's package and the library never imports it.
"""
from .cmsd_oracle import (  # noqa: F401
    Params,
    Result,
    accept_paper,
    accept_sampled,
    bf16_bits_to_f64,
    bonus_token,
    confidence,
    confidence_verify,
    decode_sim_sequence,
    drafter_signals,
    log_softmax,
    logits_to_f64,
    next_draft_length,
    rank_gate,
    residual_token,
    softmax,
    tau_t,
    two_level_race,
    unified_confidence,
    verify,
    verify_sequence,
)
from . import philox  # noqa: F401
from .lmhead import lm_head_confidence, lm_head_logits, signal_error_bound  # noqa: F401
