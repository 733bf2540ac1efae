"""GB300 (sm_103a) library for the Fusion staged token-adaptation step
(merge -> exit-check -> prune -> compact) of Vision Transformers.

The computation lives in libfusion.so (hand-written CUDA, C ABI in
include/fusion.h).  This package is its Python binding: the C functions under
the same names, plus buffer plumbing in :mod:`.runner`.
"""
from ._binding import (  # noqa: F401
    EXPORTED,
    FUSION_BF16,
    FUSION_DEV_BAD_BATCH,
    FUSION_DEV_BAD_IDS,
    FUSION_DEV_BAD_OFFSETS,
    FUSION_DEV_INTERNAL,
    FUSION_DEV_NONFINITE,
    FUSION_DEV_TIMEOUT,
    FUSION_ERR_CUDA,
    FUSION_ERR_DTYPE,
    FUSION_ERR_INVALID_ARG,
    FUSION_ERR_SHAPE,
    FUSION_ERR_WORKSPACE,
    FUSION_F32,
    FUSION_FUSED_PLAN_MAX_BATCH,
    FUSION_MAX_DIM,
    FUSION_MAX_TOKENS,
    FUSION_OK,
    FUSION_STAGE_EXIT,
    FUSION_STAGE_MERGE,
    FUSION_STAGE_PRUNE,
    FusionError,
    check,
    exit_head,
    fusion_compact,
    fusion_exit_check,
    fusion_exit_check_noalloc,
    fusion_merge,
    fusion_merge_router,
    fusion_token_scores,
    fusion_exit_check_mlp,
    fusion_exit_mlp_workspace_size,
    mlp_head,
    FUSION_POOL_CLS,
    FUSION_POOL_SPATIAL,
    fusion_profile_next,
    fusion_prune,
    fusion_stage,
    fusion_status_string,
    fusion_version,
    fusion_workspace_size,
    load,
    ragged,
)
from .build import LIB, build  # noqa: F401
