"""fp64 CPU oracle (test infrastructure only; never imported by the product path)."""

from .budgetdraft_oracle import (  # noqa: F401
    accept_greedy,
    advance_window,
    append_view,
    attention,
    batch_advance,
    boundary_score,
    combine,
    draft_attn,
    greedy_argmax,
    select_budget,
    select_from_scores,
    spec_step,
    topk_lower_index,
    verify_attn,
    widen_bf16_bits,
    window_lse,
    window_positions,
    window_scores,
)
