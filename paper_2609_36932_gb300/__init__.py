"""GB300 kept-token GRPO path of FastRL ("Learn from the Gap", Sec. 3 and Algorithm 1).

The computation lives in libfastrl_grpo.so (hand-written CUDA for sm_103a behind the C ABI of
include/fastrl_grpo.h); `binding` marshals torch tensors into it.  `workloads` draws the seeded
synthetic inputs.  Importing the package does not load the library; the first call does.
"""
from .binding import (ArsState, GrpoError, adaptive_rollout_count, check_status, checked_build,
                      grpo_advantage, grpo_debug_checks,
                      grpo_ars_deserialize, grpo_ars_init, grpo_ars_serialize, grpo_compact,
                      grpo_gspo_loss_fwd_bwd, grpo_kernel_launches, grpo_last_error,
                      grpo_lmhead_dlogits_stride, grpo_lmhead_grad,
                      grpo_lmhead_gspo_loss_fwd_bwd, grpo_lmhead_logp_fwd, grpo_lmhead_loss_fwd_bwd, grpo_lmhead_tune,
                      grpo_logp_fwd, grpo_loss_fwd_bwd, grpo_loss_fwd_bwd_dev,
                      grpo_loss_fwd_bwd_noalloc, grpo_loss_tune, grpo_prune, grpo_sum_f64,
                      grpo_upload_kept, lib, library_path, version)

__all__ = ["ArsState", "GrpoError", "adaptive_rollout_count", "check_status", "checked_build",
           "grpo_advantage", "grpo_debug_checks",
           "grpo_ars_deserialize", "grpo_ars_init", "grpo_ars_serialize", "grpo_compact",
           "grpo_gspo_loss_fwd_bwd", "grpo_kernel_launches", "grpo_last_error",
           "grpo_lmhead_dlogits_stride", "grpo_lmhead_grad", "grpo_lmhead_gspo_loss_fwd_bwd",
           "grpo_lmhead_logp_fwd",
           "grpo_lmhead_loss_fwd_bwd", "grpo_lmhead_tune", "grpo_logp_fwd", "grpo_loss_fwd_bwd",
           "grpo_loss_fwd_bwd_dev", "grpo_loss_fwd_bwd_noalloc", "grpo_loss_tune", "grpo_prune",
           "grpo_sum_f64", "grpo_upload_kept", "lib", "library_path", "version"]
