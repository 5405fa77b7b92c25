"""Float64 CPU oracle of the GRPO hot path (test infrastructure only).

Imported by tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg;
never by the library.  See grpo_oracle for the definitions it follows.
"""
from .grpo_oracle import (  # noqa: F401
    adamw_step, as_f64, gumbel_noise, sample_tokens, dH_rows, dW_rows, group_advantages, grpo_loss, logp_coef, loss_fwd_bwd,
    nucleus, sample_tokens_top_p, target_logits, token_advantages, token_logprobs, token_terms, token_weights, widen_bf16,
)
