"""GB300-native trainer -> rollout weight synchronisation hot path.

RobustRL (arXiv 2512.22492) Section 5.2.1: reshard the trainer's weights to
the rollout's sharding and copy them, one layer after another, into a transfer buffer;
Section 5.2.2: a rollout that reconnects after a failure pulls (part of) that
buffer again.  This package is the on-GPU part of that route for one GB300:
a C-ABI CUDA library (``include/rr.h``, ``csrc/``) and its Python binding.
"""
from .rr import (Block, DstLayout, DstTensor, Param, Plan, PlanOptions, Pointers, RRError,
                 SrcLayout,
                 rr_clear_range, rr_pack, rr_pack_range, rr_plan_check, rr_plan_create,
                 rr_plan_selftest_wait, rr_status_str, rr_unpack,
                 rr_unpack_range, rr_unpack_verify, rr_unpack_verify_async, rr_verify,
                 rr_verify_noalloc,
                 rr_verify_range)
from .layouts import qwen3_layer_units, qwen3_manifest, qwen3_rollout, qwen3_sync

__all__ = ["Block", "DstLayout", "DstTensor", "Param", "Plan", "PlanOptions", "Pointers",
           "RRError",
           "SrcLayout", "rr_pack", "rr_plan_create", "rr_status_str", "rr_unpack", "rr_verify",
           "rr_pack_range", "rr_unpack_range", "rr_verify_range", "rr_clear_range",
           "rr_unpack_verify", "rr_unpack_verify_async", "rr_plan_check", "rr_plan_selftest_wait", "rr_verify_noalloc",
           "qwen3_layer_units", "qwen3_manifest", "qwen3_rollout", "qwen3_sync"]
