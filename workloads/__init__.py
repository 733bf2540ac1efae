"""Seeded synthetic inputs shaped like the paper's DeiT/ViT workloads.

This package only draws random inputs and rounds them to the storage dtype.
It holds none of the merge / exit / prune / compact arithmetic, so it can serve
both the CPU oracle and the CUDA path without coupling them.
"""
from .synth import (  # noqa: F401
    CONFIGS,
    Batch,
    POOL_CLS,
    POOL_SPATIAL,
    Head,
    MlpHead,
    RouterSpec,
    ScoreHeadSpec,
    StageSpec,
    Workload,
    bf16_bits_to_f32,
    f32_to_bf16_bits,
    make_mlp_head,
    make_router,
    make_score_head,
    make_workload,
)
