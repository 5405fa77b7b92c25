"""GB300-native (sm_103a) GRPO hot path: advantages, LM-head log-probs, clipped
objective with KL penalty, and its backward to H and W (Section 3.3, Eq. 1-2).

The compute lives in libgrpo.so (C ABI in include/grpo.h); this package is
its ctypes binding plus the in-tree build script.
"""
from .binding import (  # noqa: F401
    GRPO_ERR_CAPACITY, GRPO_ERR_CUDA, GRPO_ERR_DEVICE_CHECK, GRPO_ERR_INVALID_ARG, GRPO_ERR_TIMEOUT,
    GRPO_ERR_UNSUPPORTED, GRPO_ERR_WORKSPACE, GRPO_MAX_HEADS, GRPO_OK, GRPO_WS_LOGPROBS, GRPO_WS_LOGPROBS_HEADS,
    GRPO_WS_LOSS, GRPO_WS_LOSS_LOGITS, GRPO_WS_SAMPLE, GRPO_WS_SAMPLE_TOP_P, LIB_PATH, SIGNATURES, GrpoError,
    adamw_step, check_device_status, group_advantages, gumbel_noise, load, loss_fwd_bwd, loss_fwd_bwd_adamw,
    loss_plan, loss_workspace, sample_tokens, sample_tokens_top_p, status_string, token_logprobs,
    token_logprobs_heads, vocab_chunk_cols, workspace, workspace_bytes, workspace_bytes_rows,
)
