"""Every float32 bit pattern through the pack kernels, against the oracle's cast
(to bfloat16, and to float16 for a float16 rollout).

The source is one fp32 parameter of 2^32 elements ([65536, 65536], 16 GiB)
whose element i holds the bit pattern i, in 7 flat shards (so shard cuts fall
inside rows).  Its rollout tensor is the whole parameter, so bucket stream
byte 2i holds the cast of pattern i: every rounding tie of both parities,
every subnormal, overflow into infinity, both infinities and every NaN
payload.  Each pack kernel writes it:

* the bulk-copy engine (device source),
* the register path (RR_ENGINE_REGISTERS),
* the register path reading the source from pinned host memory (HOST_SRC),

and every bucket byte and checksum is compared with the oracle's cast of the
same patterns and the oracle's word sum (the bf16 rollout image of RobustRL
Section 5.2.1 step 1, with the checksum of Section 5.2.2).  All 2^16 bf16
patterns go through the identity path of the same three kernels.
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

N = 1 << 32
CHUNK = 1 << 26                  # patterns per comparison chunk (128 MiB of bf16)
BUCKET = 256 << 20               # two chunks per bucket


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def plan_of(desc, **opts):
    m, s, d = U.to_product(desc)
    return H.make_plan(m, s, d, desc["bucket_bytes"], **opts)


@pytest.mark.parametrize("dst", ["bf16", "f16"])
def test_every_float32_pattern(dst):
    desc = dict(params=[("w", (65536, 65536), 4)], tensors=[("w", 0, [(0, 0, 65536, 0, 65536)])],
                tp=1, sharding="flat", n_shards=7, bucket_bytes=BUCKET, align_bytes=16,
                tensor_align=256, seed=1, specials=False, dst_dtype=dst)
    cast = oracle.rne_f16 if dst == "f16" else oracle.rne_bf16
    auto = plan_of(desc)
    regs = plan_of(desc, engine="registers")
    assert auto.n_buckets == regs.n_buckets == N * 2 // BUCKET
    dev = H.alloc(auto, with_dst=False)
    words = dev.flat.view(torch.int32)
    assert words.numel() >= N
    step = 1 << 28
    for s in range(0, N, step):     # element i holds the bit pattern i
        words[s:s + step].copy_(
            torch.arange(s, s + step, dtype=torch.int64, device="cuda").view(torch.int32)[0::2])
    host = torch.empty(dev.flat.numel(), dtype=torch.uint8, pin_memory=True)
    host.copy_(dev.flat)
    runs = {"bulk": dev,
            "registers": H.alloc(regs, flat=dev.flat, with_dst=False),
            "host source": H.alloc(auto, flat=host, with_dst=False)}
    H.pack(runs["bulk"])
    H.pack(runs["registers"])
    H.pack(runs["host source"])
    torch.cuda.synchronize()
    rr.rr_plan_check(auto)
    rr.rr_plan_check(regs)
    for name, buf in runs.items():
        assert buf.bucket_store.shape[1] == BUCKET, name

    def one(c):
        pats = np.arange(CHUNK, dtype=np.uint32) + np.uint32(c * CHUNK)
        want = cast(pats).view(np.uint8)
        b, off = divmod(c * CHUNK * 2, BUCKET)
        for name, buf in runs.items():
            got = buf.bucket_store[b, off:off + CHUNK * 2].cpu().numpy()
            if not np.array_equal(got, want):
                i = int(np.flatnonzero(got != want)[0]) // 2
                raise AssertionError(f"{name}: pattern {c * CHUNK + i:#010x} cast to "
                                     f"{got[2 * i:2 * i + 2].view(np.uint16)[0]:#06x}, oracle "
                                     f"{want[2 * i:2 * i + 2].view(np.uint16)[0]:#06x}")
        return b, oracle.checksum(want)

    with ThreadPoolExecutor(max_workers=min(4, os.cpu_count() or 1)) as ex:
        parts = list(ex.map(one, range(N // CHUNK)))
    want_cs = np.zeros(auto.n_buckets, np.uint64)
    for b, cs in parts:                       # a word sum is additive over aligned pieces
        want_cs[b] = np.uint64((int(want_cs[b]) + cs) % (1 << 64))
    for name, buf in runs.items():
        np.testing.assert_array_equal(H.checksums_host(buf), want_cs, err_msg=name)


@pytest.mark.parametrize("dst", ["bf16", "f16"])
@pytest.mark.parametrize("where", ["bulk", "registers", "host source"])
def test_every_bfloat16_pattern(where, dst):
    """bf16 -> bf16 is a bit copy, NaN payloads included; bf16 -> f16 widens and
    rounds: all 2^16 patterns, in 3 flat shards and 8 KiB buckets, against the
    oracle's pack."""
    desc = dict(params=[("v", (256, 256), 2)], tensors=[("v", 0, [(0, 0, 256, 0, 256)])],
                tp=1, sharding="flat", n_shards=3, bucket_bytes=8192, align_bytes=16,
                tensor_align=256, seed=1, specials=False, dst_dtype=dst)
    plan = plan_of(desc, engine="registers" if where == "registers" else "auto")
    L = U.to_oracle(desc)
    starts = H.source_offsets(plan)
    flat = np.zeros(starts[-1], np.uint8)
    flat[:1 << 17] = np.arange(1 << 16, dtype=np.uint16).view(np.uint8)
    shards = [flat[starts[i]:starts[i + 1]] for i in range(len(starts) - 1)]
    if where == "host source":
        buf = H.alloc(plan, flat=torch.from_numpy(flat.copy()).pin_memory())
    else:
        buf = H.alloc(plan)
        H.fill_from_host(buf, shards)
    H.pack(buf)
    torch.cuda.synchronize()
    want, want_cs = L.pack(oracle.Source(shards=shards))
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
    stream = want.reshape(-1)[:1 << 17].view(np.uint16)
    patterns = np.arange(1 << 16, dtype=np.uint32)
    if dst == "bf16":
        np.testing.assert_array_equal(stream, patterns.astype(np.uint16))
    else:
        np.testing.assert_array_equal(stream, oracle.rne_f16(patterns << 16))
