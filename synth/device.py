"""Device-side inputs and buffers for one weight sync (torch allocations).

The benchmark, the smoke check and the GPU tests take their buffers from here:
the trainer's source shards (filled by the seeded device generator, or copied
from host shards), one equally spaced block of buckets or separately allocated
ones, the checksum array and the rollout tensors.  Sizes come from a plan
object's geometry (``source_buffer_bytes``, ``n_buckets``, ``bucket_bytes``,
``tensor_numel``, sharding and offsets); this module imports neither the
library nor the oracle and holds none of the method's arithmetic.
"""
from __future__ import annotations

from dataclasses import dataclass
from typing import List, Optional

import numpy as np
import torch

from . import fill_dev


@dataclass
class SyncBuffers:
    plan: object
    flat: torch.Tensor                 # every source buffer, 16-byte starts, uint8
    shards: List[int]                  # device pointers into flat
    bucket_store: torch.Tensor         # [n_buckets, row >= bucket_bytes] uint8 (uniform layout)
    buckets: list                      # what is passed as the bucket array
    checksums: torch.Tensor            # [n_buckets] int64 (uint64 bits)
    dst: List[torch.Tensor]            # one int16 tensor per destination tensor


def source_offsets(plan) -> List[int]:
    """Byte offset of every source buffer in one allocation (each at a 16-byte
    start), then the total.  Shards of one FlatParameter follow one another."""
    out, off = [], 0
    for nb in plan.source_buffer_bytes:
        out.append(off)
        off += (nb + 15) // 16 * 16
    return out + [off]


def alloc(plan, separate_buckets: bool = False, poison: Optional[int] = 0xAB,
          with_dst: bool = True, flat: Optional[torch.Tensor] = None,
          device: str = "cuda") -> SyncBuffers:
    """Every buffer of one sync on `device`.  `poison` fills buckets and tensors
    (None: left uninitialised) so that unwritten bytes show; separately
    allocated buckets are shuffled so that their pointers are not equally
    spaced (the pointer-table launch shape)."""
    dev = torch.device(device)
    starts = source_offsets(plan)
    if flat is None:
        flat = torch.zeros(starts[-1], dtype=torch.uint8, device=dev)
    assert flat.numel() == starts[-1]
    base = flat.data_ptr()
    shards = [base + o for o in starts[:-1]]
    if separate_buckets:
        bl = [torch.empty(plan.bucket_bytes, dtype=torch.uint8, device=dev)
              for _ in range(plan.n_buckets)]
        if poison is not None:
            for b in bl:
                b.fill_(poison)
        order = np.random.default_rng(plan.n_buckets).permutation(len(bl))
        bl = [bl[i] for i in order]
        buckets = bl
        bucket_store = bl
    else:
        # One allocation; rows padded to 16 bytes so every bucket is 16-byte aligned.
        row = (plan.bucket_bytes + 15) // 16 * 16
        bucket_store = torch.empty((plan.n_buckets, row), dtype=torch.uint8, device=dev)
        if poison is not None:
            bucket_store.fill_(poison)
        buckets = bucket_store[:, :plan.bucket_bytes]
    checksums = torch.zeros(max(1, plan.n_buckets), dtype=torch.int64, device=dev)
    dst = [torch.empty(max(1, n), dtype=torch.int16, device=dev)
           for n in plan.tensor_numel] if with_dst else []
    if poison is not None:
        for d in dst:
            d.fill_(0x5A5A)
    return SyncBuffers(plan, flat, shards, bucket_store, buckets, checksums, dst)


def fill_from_host(buf: SyncBuffers, host_shards) -> None:
    """Copies host shard arrays (in source-buffer order) into the source block."""
    host = np.concatenate([np.asarray(s, np.uint8) for s in host_shards])
    assert host.size == buf.flat.numel()
    buf.flat.copy_(torch.from_numpy(host))


def _flat_offsets(manifest, align):
    """Flat-layout offsets: generated values are indexed by them under any sharding."""
    offs, off = [], 0
    for p in manifest:
        es = 4 if p.dtype == "f32" else 2
        a = max(align, es)
        off = (off + a - 1) // a * a
        offs.append(off)
        off += (int(np.prod(p.shape)) if len(p.shape) else 1) * es
    return offs


def fill_with_generator(buf: SyncBuffers, manifest, seed: int, specials: bool,
                        stream: int = 0) -> None:
    """Device generator, one launch per parameter (per shard for a row-sharded
    trainer) at the plan's offsets; values are indexed by the flat layout, so a
    seed gives the same parameters under every sharding."""
    plan = buf.plan
    base = buf.flat.data_ptr()
    if plan.sharding == "units":
        # Each unit's shards are adjacent, so the unit is one flat buffer.
        starts = source_offsets(plan)
        per_unit = plan.n_shards // (max(plan.units) + 1)
        flat = _flat_offsets(manifest, plan.align_bytes)
        for p, local, f, u in zip(manifest, plan.param_flat_offset, flat, plan.units):
            es = 4 if p.dtype == "f32" else 2
            n = int(np.prod(p.shape)) if len(p.shape) else 1
            fill_dev(base + starts[u * per_unit] + local, n, es, seed, first_idx=f // es,
                     specials=specials, stream=stream)
        return
    if plan.sharding == "flat":
        for p, off in zip(manifest, plan.param_flat_offset):
            es = 4 if p.dtype == "f32" else 2
            n = int(np.prod(p.shape)) if len(p.shape) else 1
            fill_dev(base + off, n, es, seed, first_idx=off // es, specials=specials,
                     stream=stream)
        return
    S = plan.shard_bytes
    flat = _flat_offsets(manifest, plan.align_bytes)
    for p, local, f in zip(manifest, plan.param_flat_offset, flat):
        es = 4 if p.dtype == "f32" else 2
        rows = p.shape[0] if len(p.shape) else 1
        cols = int(np.prod(p.shape[1:])) if len(p.shape) > 1 else 1
        c = -(-rows // plan.n_shards)
        for s in range(plan.n_shards):
            r0, r1 = s * c, min((s + 1) * c, rows)
            if r1 > r0:
                fill_dev(base + s * S + local, (r1 - r0) * cols, es, seed,
                         first_idx=f // es + r0 * cols, specials=specials, stream=stream)


def bucket_list(buf: SyncBuffers):
    if isinstance(buf.buckets, torch.Tensor):
        return [buf.buckets[i] for i in range(buf.buckets.shape[0])]
    return list(buf.buckets)
