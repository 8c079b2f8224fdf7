"""Seeded synthetic inputs for the weight-sync path: workload shapes and values.

Input generation only.  This module holds none of the method's arithmetic: it
names the model shapes of the five workloads (plus full-size variants and
scaled-down test shapes)
and draws parameter values from a counter-based generator that is defined
once and implemented twice, on the host (``synth_host.c``) and on the device
(``synth_dev.cu``).  Both the oracle and the CUDA path take their inputs from
here; neither imports the other.

The paper trains Qwen3-8B/32B/235B-A22B (Section 7.1, "Testbed"); no weights
are available here and none are needed: only the shapes and the value
distribution matter to a reshard/cast/pack, so values are drawn from
approximately N(0, 0.02) (see ``synth_host.c`` for the exact definition).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass, replace
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_HOST_SO = os.path.join(_BUILD, "libsynth_host.so")
_DEV_SO = os.path.join(_BUILD, "libsynth_dev.so")

MiB = 1 << 20


# --------------------------------------------------------------------------
# Workload shapes
# --------------------------------------------------------------------------

@dataclass(frozen=True)
class ModelShape:
    """Decoder shape in the Qwen3 family (dense or MoE)."""

    name: str
    layers: int
    hidden: int
    n_q: int            # query heads
    n_kv: int           # key/value heads
    head_dim: int
    intermediate: int   # dense MLP width (0 for MoE)
    vocab: int
    tied: bool          # lm_head shares the embedding
    n_experts: int = 0
    moe_intermediate: int = 0

    @property
    def moe(self) -> bool:
        return self.n_experts > 0


@dataclass(frozen=True)
class Workload:
    """One weight-sync problem: model shape, trainer shards, rollout TP, buckets, seed."""

    name: str
    shape: ModelShape
    src_dtype: str      # "f32" or "bf16": dtype of the trainer's parameter state
    n_shards: int       # flat FSDP-style shards
    tp: int             # rollout tensor-parallel degree
    bucket_bytes: int
    seed: int
    specials: bool = False   # inject ~1% special bit patterns
    sharding: str = "flat"   # "flat" (one FSDP1 FlatParameter), "rows" (FSDP2 dim-0), or
                             # "units" (FSDP1, one FlatParameter per decoder layer + root)
    ep: bool = False         # rollout experts split whole over the ranks (expert parallel)
    dst_dtype: str = "bf16"  # the rollout's 16-bit element type: "bf16" or "f16"

    @property
    def src_elem_bytes(self) -> int:
        return 4 if self.src_dtype == "f32" else 2

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


TINY = ModelShape("tiny", layers=2, hidden=256, n_q=4, n_kv=2, head_dim=64,
                  intermediate=688, vocab=1024, tied=False)
QWEN3_0_6B = ModelShape("qwen3-0.6b", layers=28, hidden=1024, n_q=16, n_kv=8, head_dim=128,
                        intermediate=3072, vocab=151936, tied=True)
QWEN3_8B = ModelShape("qwen3-8b", layers=36, hidden=4096, n_q=32, n_kv=8, head_dim=128,
                      intermediate=12288, vocab=151936, tied=False)
QWEN3_32B = ModelShape("qwen3-32b", layers=64, hidden=5120, n_q=64, n_kv=8, head_dim=128,
                       intermediate=25600, vocab=151936, tied=False)
QWEN3_30B_A3B = ModelShape("qwen3-30b-a3b", layers=48, hidden=2048, n_q=32, n_kv=4,
                           head_dim=128, intermediate=0, vocab=151936, tied=False,
                           n_experts=128, moe_intermediate=768)

# The five workloads.  "MB" in their descriptions is read as MiB.
WORKLOADS = {
    "tiny": Workload("tiny", TINY, "f32", n_shards=1, tp=1, bucket_bytes=256 * 1024, seed=1,
                     specials=True),
    "qwen3-0.6b": Workload("qwen3-0.6b", QWEN3_0_6B, "f32", n_shards=8, tp=1,
                           bucket_bytes=32 * MiB, seed=2),
    "qwen3-8b": Workload("qwen3-8b", QWEN3_8B, "f32", n_shards=8, tp=1,
                         bucket_bytes=128 * MiB, seed=3),
    "qwen3-8b-tp4": Workload("qwen3-8b-tp4", QWEN3_8B, "f32", n_shards=8, tp=4,
                             bucket_bytes=128 * MiB, seed=4),
    "qwen3-30b-a3b": Workload("qwen3-30b-a3b", QWEN3_30B_A3B, "bf16", n_shards=8, tp=1,
                              bucket_bytes=256 * MiB, seed=5),
}

# Bucket sizes swept on the TP=4 workload.
TP4_BUCKET_SWEEP = [s * MiB for s in (4, 8, 16, 32, 64, 128, 256, 512)]

# Scaled-down shapes for tests: same structure, sizes the oracle finishes in seconds.
TINY_MOE = ModelShape("tiny-moe", layers=2, hidden=128, n_q=4, n_kv=2, head_dim=32,
                      intermediate=0, vocab=512, tied=False, n_experts=8, moe_intermediate=96)
TINY_TIED = replace(TINY, name="tiny-tied", tied=True)
ODD = ModelShape("odd", layers=2, hidden=257, n_q=2, n_kv=1, head_dim=36,
                 intermediate=689, vocab=301, tied=False)

TEST_WORKLOADS = {
    "tiny-tp4": Workload("tiny-tp4", TINY, "f32", n_shards=8, tp=4, bucket_bytes=64 * 1024,
                         seed=14, specials=True),
    "tiny-tied": Workload("tiny-tied", TINY_TIED, "f32", n_shards=8, tp=1,
                          bucket_bytes=96 * 1024, seed=12),
    "tiny-moe": Workload("tiny-moe", TINY_MOE, "bf16", n_shards=8, tp=1,
                         bucket_bytes=128 * 1024, seed=15),
    "tiny-moe-tp2": Workload("tiny-moe-tp2", TINY_MOE, "bf16", n_shards=3, tp=2,
                             bucket_bytes=40 * 1024, seed=16),
    "tiny-moe-f32": Workload("tiny-moe-f32", TINY_MOE, "f32", n_shards=5, tp=2,
                             bucket_bytes=24 * 1024, seed=17, specials=True),
    # bf16 trainer state carrying the special bit patterns (signalling NaNs must
    # pass through a bf16 -> bf16 copy untouched).
    "tiny-moe-bf16-specials": Workload("tiny-moe-bf16-specials", TINY_MOE, "bf16", n_shards=4,
                                       tp=2, bucket_bytes=32 * 1024, seed=21, specials=True),
    # FSDP2-style (each parameter cut on dim 0) trainers; uneven chunks.
    "tiny-fsdp2": Workload("tiny-fsdp2", TINY, "f32", n_shards=3, tp=2, bucket_bytes=48 * 1024,
                           seed=18, specials=True, sharding="rows"),
    # TP above the KV head count: KV heads replicated over ranks.
    "tiny-moe-kvrep": Workload("tiny-moe-kvrep", TINY_MOE, "bf16", n_shards=6, tp=4,
                               bucket_bytes=32 * 1024, seed=19, sharding="rows"),
    "tiny-kvrep-f32": Workload("tiny-kvrep-f32", TINY, "f32", n_shards=8, tp=8,
                               bucket_bytes=16 * 1024, seed=20, specials=True),
    # FSDP1 wrapping every decoder layer: one FlatParameter per layer plus the root's.
    "tiny-units": Workload("tiny-units", TINY, "f32", n_shards=3, tp=2, bucket_bytes=48 * 1024,
                           seed=22, specials=True, sharding="units"),
    # Expert-parallel rollouts: every rank holds whole experts.
    "tiny-moe-ep4": Workload("tiny-moe-ep4", TINY_MOE, "f32", n_shards=8, tp=4,
                             bucket_bytes=24 * 1024, seed=23, specials=True, ep=True),
    "tiny-moe-units-ep2": Workload("tiny-moe-units-ep2", TINY_MOE, "bf16", n_shards=5, tp=2,
                                   bucket_bytes=32 * 1024, seed=24, sharding="units", ep=True),
}

# Full-size variants beyond the five workloads: the paper's own trainer sharding
# (FSDP2, Section 7.1) and its rollout TP of 8.
EXTRA_WORKLOADS = {
    "qwen3-8b-fsdp2-tp8": Workload("qwen3-8b-fsdp2-tp8", QWEN3_8B, "f32", n_shards=8, tp=8,
                                   bucket_bytes=128 * MiB, seed=6, sharding="rows"),
    "qwen3-30b-a3b-fsdp2-tp8": Workload("qwen3-30b-a3b-fsdp2-tp8", QWEN3_30B_A3B, "bf16",
                                        n_shards=8, tp=8, bucket_bytes=256 * MiB, seed=7,
                                        sharding="rows"),
    # Per-layer FSDP1 units (the common FSDP1 wrapping) and an expert-parallel rollout.
    "qwen3-8b-units": Workload("qwen3-8b-units", QWEN3_8B, "f32", n_shards=8, tp=1,
                               bucket_bytes=128 * MiB, seed=8, sharding="units"),
    "qwen3-30b-a3b-fsdp2-ep8": Workload("qwen3-30b-a3b-fsdp2-ep8", QWEN3_30B_A3B, "bf16",
                                        n_shards=8, tp=8, bucket_bytes=256 * MiB, seed=9,
                                        sharding="rows", ep=True),
    # The paper's Qwen3-32B with its FSDP2 trainer and TP=8 rollout: the largest
    # of its models whose whole sync fits one GPU (131 GB of fp32 source, 67 GB
    # of buckets and 66 GB of rollout tensors: 245 GiB).
    "qwen3-32b-fsdp2-tp8": Workload("qwen3-32b-fsdp2-tp8", QWEN3_32B, "f32", n_shards=8, tp=8,
                                    bucket_bytes=128 * MiB, seed=10, sharding="rows"),
}


# --------------------------------------------------------------------------
# Build
# --------------------------------------------------------------------------

def _stale(out: str, srcs) -> bool:
    if not os.path.exists(out):
        return True
    t = os.path.getmtime(out)
    return any(os.path.getmtime(s) > t for s in srcs)


def build_host() -> str:
    srcs = [os.path.join(_HERE, "synth_host.c"), os.path.join(_HERE, "synth_specials.h")]
    if _stale(_HOST_SO, srcs):
        os.makedirs(_BUILD, exist_ok=True)
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off",
                               "-o", _HOST_SO, srcs[0]])
    return _HOST_SO


def build_dev() -> str:
    srcs = [os.path.join(_HERE, "synth_dev.cu"), os.path.join(_HERE, "synth_specials.h")]
    if _stale(_DEV_SO, srcs):
        os.makedirs(_BUILD, exist_ok=True)
        subprocess.check_call(["nvcc", "-O3", "-std=c++17", "-shared", "-Xcompiler", "-fPIC",
                               "-gencode", "arch=compute_103a,code=sm_103a", "-lineinfo",
                               "-fmad=false", "-o", _DEV_SO, srcs[0]])
    return _DEV_SO


def build() -> None:
    build_host()
    build_dev()


# --------------------------------------------------------------------------
# Host generator
# --------------------------------------------------------------------------

_host_lib: Optional[ctypes.CDLL] = None
_dev_lib: Optional[ctypes.CDLL] = None


class SynthCtx(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("specials", ctypes.c_int32)]


def host_lib() -> ctypes.CDLL:
    global _host_lib
    if _host_lib is None:
        lib = ctypes.CDLL(build_host())
        lib.synth_fill_host.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int,
                                        ctypes.c_uint64, ctypes.c_int64, ctypes.c_int]
        lib.synth_fill_host.restype = None
        lib.synth_gather_host.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                          ctypes.c_int, ctypes.c_uint64, ctypes.c_int]
        lib.synth_gather_host.restype = None
        lib.synth_splitmix64.argtypes = [ctypes.c_uint64]
        lib.synth_splitmix64.restype = ctypes.c_uint64
        lib.synth_f32_bits.argtypes = [ctypes.c_uint64, ctypes.c_int64, ctypes.c_int]
        lib.synth_f32_bits.restype = ctypes.c_uint32
        lib.synth_n_special.restype = ctypes.c_int
        lib.synth_special_table.argtypes = [ctypes.c_void_p]
        lib.synth_value_fn.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32]
        lib.synth_value_fn.restype = ctypes.c_uint32
        _host_lib = lib
    return _host_lib


def values_host(n: int, elem_bytes: int, seed: int, first_idx: int = 0,
                specials: bool = False) -> np.ndarray:
    """Bit patterns of elements first_idx..first_idx+n-1 (uint32 for fp32, uint16 for bf16)."""
    out = np.empty(n, dtype=np.uint32 if elem_bytes == 4 else np.uint16)
    if n:
        host_lib().synth_fill_host(out.ctypes.data, n, elem_bytes, seed, first_idx, int(specials))
    return out


def gather_host(idx: np.ndarray, elem_bytes: int, seed: int, specials: bool = False) -> np.ndarray:
    """Bit patterns at arbitrary element indices."""
    idx = np.ascontiguousarray(idx, dtype=np.int64)
    out = np.empty(idx.size, dtype=np.uint32 if elem_bytes == 4 else np.uint16)
    if idx.size:
        host_lib().synth_gather_host(out.ctypes.data, idx.ctypes.data, idx.size, elem_bytes,
                                     seed, int(specials))
    return out


def special_table() -> np.ndarray:
    lib = host_lib()
    out = np.empty(lib.synth_n_special(), dtype=np.uint32)
    lib.synth_special_table(out.ctypes.data)
    return out


def value_fn_ptr() -> int:
    """Address of the C function ``uint32_t f(const void* ctx, int64_t idx, int32_t elem_bytes)``."""
    return ctypes.cast(host_lib().synth_value_fn, ctypes.c_void_p).value


# --------------------------------------------------------------------------
# Device generator
# --------------------------------------------------------------------------

def dev_lib() -> ctypes.CDLL:
    global _dev_lib
    if _dev_lib is None:
        lib = ctypes.CDLL(build_dev())
        lib.synth_fill_dev.argtypes = [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int,
                                       ctypes.c_uint64, ctypes.c_int64, ctypes.c_int,
                                       ctypes.c_void_p]
        lib.synth_fill_dev.restype = ctypes.c_int
        lib.synth_gather_dev.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64,
                                         ctypes.c_int, ctypes.c_uint64, ctypes.c_int,
                                         ctypes.c_void_p]
        lib.synth_gather_dev.restype = ctypes.c_int
        _dev_lib = lib
    return _dev_lib


def fill_dev(ptr: int, n: int, elem_bytes: int, seed: int, first_idx: int = 0,
             specials: bool = False, stream: int = 0) -> None:
    """Fill n elements at device address ptr with the values of first_idx.. (asynchronous)."""
    rc = dev_lib().synth_fill_dev(ptr, n, elem_bytes, seed, first_idx, int(specials), stream)
    if rc != 0:
        raise RuntimeError(f"synth_fill_dev failed with code {rc}")


def gather_dev(out_ptr: int, idx_ptr: int, n: int, elem_bytes: int, seed: int,
               specials: bool = False, stream: int = 0) -> None:
    rc = dev_lib().synth_gather_dev(out_ptr, idx_ptr, n, elem_bytes, seed, int(specials), stream)
    if rc != 0:
        raise RuntimeError(f"synth_gather_dev failed with code {rc}")
