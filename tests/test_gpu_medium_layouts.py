"""GPU parity on medium random layouts: odd shapes at the scale where buckets
hold many work items, against the oracle bit for bit.

``_util.random_medium_layout`` draws up to eight parameters of up to about
1500 x 3000 elements (fp32 and bf16, some 1-D), cut for TP = 1, 2, 3, 4 or 8
the ways a rollout cuts a model: rows split over the ranks (long contiguous
runs, the bulk engine's TMA copies), columns split over the ranks (row-parallel
slices: fan-out groups when the slices are 16-byte aligned multiples of 8
elements, plain strided items otherwise), replicated, or fused from two
parameters.  Trainers are flat FSDP1 shards, FSDP2 rows or per-module units,
one to eight ranks; buckets run from 64 KiB to 4 MiB, some of them 8 or 16
bytes past a power of two.  Each case moves a few to about 25 MB, so several
work units share each bucket and the claimed tails and fan-out heads are all
reached.

Every seed runs one sync (RobustRL Section 5.2.1 steps 1-2, checked as in
Section 5.2.2): rr_pack, then the verifying unpack into poisoned tensors (the
blocking form, or the stream-ordered one through pointer tables as the
benchmark calls it), then a plain rr_unpack into freshly poisoned tensors and
an rr_pack_range over three ranges into fresh buckets.  Buckets, checksums and
tensors must equal the oracle's after each.  The seeds rotate through float16
and bf16 rollouts, both engines, sources in pinned host memory and separately
allocated buckets.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

SEEDS = 40


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def options(seed):
    return dict(dst="f16" if seed % 2 else "bf16",
                engine="registers" if seed % 4 == 3 else "auto",
                host_source=seed % 5 == 1,
                separate=seed % 3 == 2,
                stream_ordered=seed % 2 == 0)


def poison_tensors(buf):
    for d in buf.dst:
        d.fill_(0x5A5A)


@pytest.mark.parametrize("seed", range(SEEDS))
def test_medium_random_layout(seed):
    o = options(seed)
    desc = U.random_medium_layout(seed)
    desc["dst_dtype"] = o["dst"]
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], engine=o["engine"])
    shards = L.host_shards(desc["seed"], desc["specials"])
    src = oracle.Source(shards=shards)
    want, want_cs = L.pack(src)
    want_t = [L.reshard_tensor(src, t) for t in range(len(L.tensors))]

    def check(buf, what, tensors=True):
        np.testing.assert_array_equal(H.buckets_host(buf), want, err_msg=f"{what}: buckets")
        np.testing.assert_array_equal(H.checksums_host(buf), want_cs, err_msg=f"{what}: checksums")
        if tensors:
            for t in range(plan.n_tensors):
                np.testing.assert_array_equal(H.tensor_host(buf, t), want_t[t],
                                              err_msg=f"{what}: tensor {plan.tensor_names[t]} "
                                                      f"rank {plan.tensor_ranks[t]}")

    if o["host_source"]:
        flat = torch.from_numpy(np.concatenate([np.asarray(x, np.uint8) for x in shards]))
        buf = H.alloc(plan, flat=flat.pin_memory(), separate_buckets=o["separate"])
    else:
        buf = H.alloc(plan, separate_buckets=o["separate"])
        H.fill_from_host(buf, shards)
    H.pack(buf)
    if o["stream_ordered"]:
        stream = torch.cuda.Stream()
        scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")
        result = torch.full((2,), -7, dtype=torch.int64, device="cuda")
        t_bkt = rr.Pointers(plan, "buckets", buf.buckets)
        t_dst = rr.Pointers(plan, "dst", buf.dst)
        stream.wait_stream(torch.cuda.current_stream())
        rr.rr_unpack_verify_async(plan, t_bkt, buf.checksums, t_dst, scratch, result,
                                  stream=stream)
        stream.synchronize()
        assert result.tolist() == [0, -1]
    else:
        assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    check(buf, "pack + verifying unpack")

    poison_tensors(buf)
    H.unpack(buf)
    torch.cuda.synchronize()
    check(buf, "rr_unpack")

    ranged = H.alloc(plan, flat=buf.flat, separate_buckets=not o["separate"], with_dst=False)
    n = plan.n_buckets
    cuts = sorted({0, n // 3, (2 * n) // 3, n})
    for a, b in reversed(list(zip(cuts[:-1], cuts[1:]))):
        rr.rr_pack_range(plan, a, b - a, ranged.shards, ranged.buckets, ranged.checksums)
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    check(ranged, "rr_pack_range", tensors=False)


def test_seed_options_cover_every_form():
    opts = [options(s) for s in range(SEEDS)]
    for key in ("host_source", "separate", "stream_ordered"):
        assert {o[key] for o in opts} == {False, True}
    assert {o["dst"] for o in opts} == {"bf16", "f16"}
    assert {o["engine"] for o in opts} == {"auto", "registers"}
