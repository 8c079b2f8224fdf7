"""One plan driven from several host threads at once.

include/rr.h lets a plan run concurrently on different streams, from different
threads, as long as the outputs are distinct (each launch takes its own
work-unit counter under the plan's lock; the blocking verify serialises on the
plan).  Here six threads share one plan and one source; each has its own
stream, buckets, checksums, tensors, scratch and result rows, and runs many
steps of rr_pack, the stream-ordered verifying unpack, bucket-range packs and
the blocking verify, so that launches contend for the plan's 16 counter slots
(and take the fallbacks when none is free).  Every thread's buckets,
checksums and tensors must equal the oracle's at the end (RobustRL Section
5.2.1: many rollouts pull from one trainer; Section 5.2.2: each checks what it
holds).
"""
import os
import threading
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

THREADS = 6
STEPS = 12


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    torch.cuda.synchronize()


@pytest.mark.parametrize("name", ["tiny-tp4", "qwen3-0.6b"])
def test_threads_share_a_plan(name):
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    shards = L.host_shards(desc["seed"], desc["specials"])
    src = H.alloc(plan, with_dst=False)
    H.fill_from_host(src, shards)
    torch.cuda.synchronize()
    t_src = rr.Pointers(plan, "src_shards", src.shards)
    n = plan.n_buckets

    class Worker:
        def __init__(self, k):
            self.buf = H.alloc(plan, flat=src.flat, poison=0xAB)
            self.stream = torch.cuda.Stream()
            self.scratch = torch.zeros(n + 4, dtype=torch.int64, device="cuda")
            self.results = torch.full((STEPS, 2), -7, dtype=torch.int64, device="cuda")
            self.t_bkt = rr.Pointers(plan, "buckets", self.buf.buckets)
            self.t_dst = rr.Pointers(plan, "dst", self.buf.dst)
            self.verified = []
            self.error = None
            self.k = k

        def run(self):
            try:
                st = self.stream
                for i in range(STEPS):
                    rr.rr_pack(plan, t_src, self.t_bkt, self.buf.checksums, st)
                    rr.rr_unpack_verify_async(plan, self.t_bkt, self.buf.checksums, self.t_dst,
                                              self.scratch, self.results[i], stream=st)
                    if i % 3 == self.k % 3 and n > 2:
                        a = (i + self.k) % (n - 1)
                        rr.rr_pack_range(plan, a, 1, t_src, self.t_bkt, self.buf.checksums, st)
                    if i % 4 == 0:
                        self.verified.append(rr.rr_verify(plan, self.t_bkt, self.buf.checksums,
                                                          st))
                self.stream.synchronize()
            except Exception as exc:   # reported by the main thread
                self.error = exc

    workers = [Worker(k) for k in range(THREADS)]
    torch.cuda.synchronize()
    threads = [threading.Thread(target=w.run) for w in workers]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    src_o = oracle.Source(shards=shards)
    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:   # the oracle, per bucket
        parts = list(ex.map(lambda b: L.pack(src_o, first=b, count=1), range(L.n_buckets)))
    want = np.concatenate([p[0] for p in parts])
    want_cs = np.concatenate([p[1] for p in parts]).astype(np.uint64)
    want_t = [L.unpack_tensor(want, t) for t in range(plan.n_tensors)]
    for w in workers:
        assert w.error is None, w.error
        assert w.verified == [(0, -1)] * len(w.verified)
        assert w.results.cpu().tolist() == [[0, -1]] * STEPS
        np.testing.assert_array_equal(H.buckets_host(w.buf), want, err_msg=f"thread {w.k}")
        np.testing.assert_array_equal(H.checksums_host(w.buf), want_cs, err_msg=f"thread {w.k}")
        for t in range(plan.n_tensors):
            np.testing.assert_array_equal(H.tensor_host(w.buf, t), want_t[t],
                                          err_msg=f"thread {w.k}, tensor {t}")
