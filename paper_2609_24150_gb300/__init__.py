"""Acceptance-aware draft-training losses (EAL / WTV) and GRPO acceptance reward on GB300.

A thin Python binding over the C ABI of ``libaal.so`` (declared in
``include/aal.h``).  Every function keeps the C name and only marshals
arguments: torch supplies device memory and the current CUDA stream, and all of
the arithmetic runs in the library's CUDA kernels.  There is no CPU fallback:
importing this package without the built library raises ImportError, and every
tensor argument must already live on the GPU.

Build the library with ``python -m paper_2609_24150_gb300.build``.
"""

from .aal import (  # noqa: F401
    AAL_BF16,
    AAL_BOTH,
    AAL_ERR_CUDA,
    AAL_ERR_INVALID_ARG,
    AAL_ERR_TIMEOUT,
    AAL_ERR_UNSUPPORTED,
    AAL_ERR_WORKSPACE,
    AAL_F32,
    AAL_GREEDY,
    AAL_GRPO,
    AAL_IDS,
    AAL_KL,
    AAL_MAX_K,
    AAL_NOALLOC_MAX_ROWS,
    AAL_OK,
    AAL_SAMPLED_DRAFT,
    AAL_SAMPLING,
    AAL_TV,
    AalError,
    AalGrpoProblem,
    AalProblem,
    AalRewardProblem,
    AalSeqProblem,
    aal_abi_version,
    aal_accept_reward,
    aal_accept_reward_from_loss,
    aal_accept_reward_sampled_from_loss,
    aal_accept_reward_noalloc,
    aal_check_device_status,
    aal_debug_fail_next_forward,
    aal_debug_fused_min_row_bytes,
    aal_debug_solo_windows,
    aal_grpo_from_loss,
    aal_grpo_workspace_size,
    aal_seq_grpo_from_loss,
    aal_seq_grpo_workspace_size,
    aal_loss_bwd,
    aal_loss_fwd,
    aal_loss_fwd_bwd,
    aal_reward_workspace_size,
    aal_seq_loss_bwd,
    aal_seq_loss_fwd_bwd,
    aal_seq_loss_fwd,
    aal_seq_workspace_size,
    aal_status_string,
    aal_workspace_size,
    library,
    library_path,
    loss_problem,
    grpo_problem,
    grpo_seq_problem,
    reward_problem,
    seq_problem,
)
