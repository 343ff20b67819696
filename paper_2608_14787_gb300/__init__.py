"""GB300 (sm_103a) logits-side hot path of verifier-skipping speculative
diffusion decoding (arXiv 2608.14787).

The compute runs in libsdd.so (hand-written CUDA behind the C ABI in
include/sdd.h); this package holds its build step, a ctypes binding with the
same entry-point names, and the seeded synthetic-input generators.
"""
from .binding import (  # noqa: F401
    BlockRound, Confidence, SddError, Workspace, agreement, block_pipelined, commit, confidence, confidence_buffers, confidence_noalloc,
    load, new_status,
    permutation_diagnostic, position_metrics, schedule_periodic, schedule_prefix, scorer_deep, scorer_features, scorer_workspace,
    select_rows, status_from_device, survival_mlp, test_wait_hooks, uniforms, verify_lenient, verify_strict, verify_strict_listed,
    verify_topk,
    workspace_bytes, SIG_RAW, SIG_MARGINAL, SIG_CONDITIONAL, SIG_PERIODIC, DEV_NONFINITE, DEV_BAD_TOKEN, DEV_TIMEOUT,
)
