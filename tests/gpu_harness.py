"""GPU-side test harness: device buffers for one weight sync (from
``synth.device``), runs of the library's calls and host copies of the results.

Used by the -m gpu tests.  It imports the library (the product) and ``synth``
(inputs), never the oracle.
"""
from __future__ import annotations

import numpy as np
import torch

import paper_2512_22492_gb300 as rr
from synth.device import (SyncBuffers, alloc, bucket_list, fill_from_host,  # noqa: F401
                          fill_with_generator, source_offsets)


def make_plan(manifest, src, dst, bucket_bytes, **opts):
    options = rr.PlanOptions(**opts) if opts else None
    return rr.rr_plan_create(manifest, src, dst, bucket_bytes, options)


def pack(buf: SyncBuffers, stream=None):
    rr.rr_pack(buf.plan, buf.shards, buf.buckets, buf.checksums, stream)


def unpack(buf: SyncBuffers, stream=None):
    rr.rr_unpack(buf.plan, buf.buckets, buf.dst, stream)


def verify(buf: SyncBuffers, stream=None):
    return rr.rr_verify(buf.plan, buf.buckets, buf.checksums, stream)


def buckets_host(buf: SyncBuffers, idx=None) -> np.ndarray:
    bl = bucket_list(buf)
    idx = range(len(bl)) if idx is None else idx
    return np.stack([bl[i].cpu().numpy() for i in idx]) if len(idx) else \
        np.zeros((0, buf.plan.bucket_bytes), np.uint8)


def checksums_host(buf: SyncBuffers) -> np.ndarray:
    return buf.checksums.cpu().numpy().view(np.uint64)[:buf.plan.n_buckets]


def tensor_host(buf: SyncBuffers, t: int) -> np.ndarray:
    return buf.dst[t][:buf.plan.tensor_numel[t]].cpu().numpy().view(np.uint16)


def device_word_sums(buf: SyncBuffers) -> np.ndarray:
    """Per-bucket 64-bit word sums computed with torch (wrapping int64 adds)."""
    out = []
    for b in bucket_list(buf):
        out.append(int(b.view(torch.int64).sum().item()) & ((1 << 64) - 1))
    return np.array(out, dtype=np.uint64)
