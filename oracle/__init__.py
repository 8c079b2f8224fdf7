"""CPU oracle for the weight-sync reshard / cast / pack / checksum / unpack / verify path.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference arm may import this package.  It
shares no code with the CUDA library (``paper_2512_22492_gb300``) and never
imports it; its inputs come from ``synth`` (shapes and seeded values) or from
the caller as plain host arrays.

The arithmetic lives in ``rr_oracle.c`` (plain single-threaded C, one element
at a time; its header states every definition and the paper passage it
follows).  This module is ctypes marshalling plus the oracle's own Qwen3
layout description (``qwen3.py``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import List, Optional, Sequence

import numpy as np

from . import qwen3

_HERE = os.path.dirname(os.path.abspath(__file__))
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liboracle.so")


def build() -> str:
    src = os.path.join(_HERE, "rr_oracle.c")
    if not os.path.exists(_SO) or os.path.getmtime(src) > os.path.getmtime(_SO):
        os.makedirs(_BUILD, exist_ok=True)
        subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", _SO, src])
    return _SO


class _Param(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("elem_bytes", ctypes.c_int32), ("pad_", ctypes.c_int32)]


class _Block(ctypes.Structure):
    _fields_ = [("param", ctypes.c_int32), ("pad_", ctypes.c_int32),
                ("row0", ctypes.c_int64), ("nrows", ctypes.c_int64),
                ("col0", ctypes.c_int64), ("ncols", ctypes.c_int64)]


class _Tensor(ctypes.Structure):
    _fields_ = [("rank", ctypes.c_int32), ("n_blocks", ctypes.c_int32),
                ("blocks", ctypes.POINTER(_Block))]


_P64 = ctypes.POINTER(ctypes.c_int64)


class _Layout(ctypes.Structure):
    _fields_ = [("n_params", ctypes.c_int32), ("n_shards", ctypes.c_int32),
                ("params", ctypes.POINTER(_Param)), ("align_bytes", ctypes.c_int64),
                ("n_tensors", ctypes.c_int32), ("tp", ctypes.c_int32),
                ("tensors", ctypes.POINTER(_Tensor)), ("tensor_align", ctypes.c_int64),
                ("bucket_bytes", ctypes.c_int64),
                ("param_offset", _P64), ("tensor_numel", _P64), ("tensor_offset", _P64),
                ("rank_stream_bytes", _P64), ("rank_first_bucket", _P64),
                ("flat_bytes", ctypes.c_int64), ("shard_bytes", ctypes.c_int64),
                ("sharding", ctypes.c_int32), ("pad_", ctypes.c_int32),
                ("shard_bytes_in", ctypes.c_int64), ("explicit_offset", _P64),
                ("chunk_rows", _P64), ("param_gen_base", _P64),
                ("n_units", ctypes.c_int32), ("pad2_", ctypes.c_int32),
                ("param_unit", ctypes.POINTER(ctypes.c_int32)), ("unit_shard_bytes", _P64),
                ("dst_dtype", ctypes.c_int32), ("pad3_", ctypes.c_int32)]


_VALUE_FN = ctypes.CFUNCTYPE(ctypes.c_uint32, ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32)


class _Source(ctypes.Structure):
    _fields_ = [("shards", ctypes.POINTER(ctypes.c_void_p)), ("gen", ctypes.c_void_p),
                ("gen_ctx", ctypes.c_void_p)]


_lib: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        _lib = load(build())
    return _lib


def load(path: str) -> ctypes.CDLL:
    """Load an oracle library build and declare its functions (the mutation
    tests load deliberately broken builds this way)."""
    L = ctypes.CDLL(path)
    LP = ctypes.POINTER(_Layout)
    SP = ctypes.POINTER(_Source)
    vp = ctypes.c_void_p
    L.orc_layout_compute.argtypes = [LP]
    L.orc_layout_compute.restype = ctypes.c_int
    L.orc_rne_bf16.argtypes = [ctypes.c_uint32]
    L.orc_rne_bf16.restype = ctypes.c_uint16
    L.orc_rne_bf16_array.argtypes = [vp, vp, ctypes.c_int64]
    L.orc_rne_bf16_array.restype = None
    L.orc_rne_f16_array.argtypes = [vp, vp, ctypes.c_int64]
    L.orc_rne_f16_array.restype = None
    L.orc_tensor_elements.argtypes = [LP, SP, ctypes.c_int32, ctypes.c_int64,
                                      ctypes.c_int64, vp]
    L.orc_tensor_elements.restype = ctypes.c_int
    L.orc_reshard_tensor.argtypes = [LP, SP, ctypes.c_int32, vp]
    L.orc_reshard_tensor.restype = ctypes.c_int
    L.orc_pack_bucket.argtypes = [LP, SP, ctypes.c_int64, vp]
    L.orc_pack_bucket.restype = ctypes.c_int
    L.orc_pack_range.argtypes = [LP, SP, ctypes.c_int64, ctypes.c_int64, vp, vp]
    L.orc_pack_range.restype = ctypes.c_int
    L.orc_checksum.argtypes = [vp, ctypes.c_int64]
    L.orc_checksum.restype = ctypes.c_uint64
    L.orc_unpack_tensor.argtypes = [LP, ctypes.POINTER(vp), ctypes.c_int32, vp]
    L.orc_unpack_tensor.restype = ctypes.c_int
    L.orc_unpack_elements.argtypes = [LP, ctypes.POINTER(vp), ctypes.c_int32, ctypes.c_int64,
                                      ctypes.c_int64, vp]
    L.orc_unpack_elements.restype = ctypes.c_int
    L.orc_verify.argtypes = [LP, ctypes.POINTER(vp), vp, ctypes.c_int64, ctypes.c_int64,
                             _P64]
    L.orc_verify.restype = ctypes.c_int64
    return L


def _check(rc: int, what: str) -> None:
    if rc != 0:
        raise RuntimeError(f"oracle {what} failed with code {rc}")


# ----------------------------------------------------------------------------
# Cast and checksum on their own
# ----------------------------------------------------------------------------

def rne_bf16(bits: np.ndarray) -> np.ndarray:
    """float32 bit patterns (uint32) -> bfloat16 bit patterns (uint16)."""
    a = np.ascontiguousarray(bits, dtype=np.uint32)
    out = np.empty(a.shape, dtype=np.uint16)
    lib().orc_rne_bf16_array(a.ctypes.data, out.ctypes.data, a.size)
    return out


def rne_f16(bits: np.ndarray) -> np.ndarray:
    """float32 bit patterns (uint32) -> IEEE binary16 bit patterns (uint16)."""
    a = np.ascontiguousarray(bits, dtype=np.uint32)
    out = np.empty(a.shape, dtype=np.uint16)
    lib().orc_rne_f16_array(a.ctypes.data, out.ctypes.data, a.size)
    return out


def checksum(data) -> int:
    """64-bit little-endian word-sum modulo 2^64 of a byte buffer (length % 8 == 0)."""
    a = np.ascontiguousarray(np.frombuffer(memoryview(data).cast("B"), dtype=np.uint8))
    return int(lib().orc_checksum(a.ctypes.data, a.size))


# ----------------------------------------------------------------------------
# Layout
# ----------------------------------------------------------------------------

class Source:
    """Where the oracle reads parameter values: host shard buffers or the seeded generator."""

    def __init__(self, shards: Optional[Sequence[np.ndarray]] = None,
                 seed: Optional[int] = None, specials: bool = False):
        self._keep = []
        self.c = _Source()
        if shards is not None:
            arrs = [None if s is None else np.ascontiguousarray(s).view(np.uint8) for s in shards]
            self._keep += arrs
            ptrs = (ctypes.c_void_p * len(arrs))(*[0 if a is None else a.ctypes.data
                                                   for a in arrs])
            self._keep.append(ptrs)
            self.c.shards = ctypes.cast(ptrs, ctypes.POINTER(ctypes.c_void_p))
        else:
            import synth
            ctx = synth.SynthCtx(seed=seed, specials=int(specials))
            self._keep.append(ctx)
            self.c.shards = None
            self.c.gen = synth.value_fn_ptr()
            self.c.gen_ctx = ctypes.addressof(ctx)


class Layout:
    """A weight-sync problem as the oracle sees it.

    params:  list of (name, dims, elem_bytes) in manifest order
    tensors: list of (name, rank, [(param, row0, nrows, col0, ncols), ...]) in plan order
    """

    def __init__(self, params, tensors, n_shards: int, tp: int, bucket_bytes: int,
                 align_bytes: int = 16, tensor_align: int = 256, sharding: str = "flat",
                 explicit_offsets=None, shard_bytes: int = 0, units=None,
                 dst_dtype: str = "bf16"):
        """units: with sharding="units", the unit of each parameter.
        dst_dtype: the rollout's 16-bit element type, "bf16" or "f16"."""
        self.sharding = sharding
        self.params = list(params)
        self.tensors = list(tensors)
        self.n_shards, self.tp, self.bucket_bytes = n_shards, tp, bucket_bytes
        self.align_bytes, self.tensor_align = align_bytes, tensor_align
        self.views = [qwen3._view(d) if len(d) else (1, 1) for _, d, _ in self.params]

        cp = (_Param * max(1, len(self.params)))()
        for i, ((_, dims, es), (rows, cols)) in enumerate(zip(self.params, self.views)):
            cp[i].rows, cp[i].cols, cp[i].elem_bytes = rows, cols, es
        self._blocks = []
        ct = (_Tensor * max(1, len(self.tensors)))()
        for i, (_, rank, blocks) in enumerate(self.tensors):
            cb = (_Block * max(1, len(blocks)))()
            for k, (p, r0, nr, c0, nc) in enumerate(blocks):
                cb[k].param, cb[k].row0, cb[k].nrows, cb[k].col0, cb[k].ncols = p, r0, nr, c0, nc
            self._blocks.append(cb)
            ct[i].rank, ct[i].n_blocks = rank, len(blocks)
            ct[i].blocks = ctypes.cast(cb, ctypes.POINTER(_Block))
        self._cp, self._ct = cp, ct

        self.param_offset = np.zeros(max(1, len(self.params)), np.int64)
        self.tensor_numel = np.zeros(max(1, len(self.tensors)), np.int64)
        self.tensor_offset = np.zeros(max(1, len(self.tensors)), np.int64)
        self.rank_stream_bytes = np.zeros(tp, np.int64)
        self.rank_first_bucket = np.zeros(tp + 1, np.int64)
        self.chunk_rows = np.zeros(max(1, len(self.params)), np.int64)
        self.param_gen_base = np.zeros(max(1, len(self.params)), np.int64)
        L = _Layout()
        L.n_params, L.n_shards = len(self.params), n_shards
        L.params = ctypes.cast(cp, ctypes.POINTER(_Param))
        L.align_bytes = align_bytes
        L.n_tensors, L.tp = len(self.tensors), tp
        L.tensors = ctypes.cast(ct, ctypes.POINTER(_Tensor))
        L.tensor_align, L.bucket_bytes = tensor_align, bucket_bytes
        for name in ("param_offset", "tensor_numel", "tensor_offset", "rank_stream_bytes",
                     "rank_first_bucket", "chunk_rows", "param_gen_base"):
            setattr(L, name, getattr(self, name).ctypes.data_as(_P64))
        L.sharding = {"flat": 0, "rows": 1, "tensors": 2, "units": 3}[sharding]
        self.dst_dtype = dst_dtype
        L.dst_dtype = {"bf16": 0, "f16": 1}[dst_dtype]
        L.shard_bytes_in = shard_bytes
        self.units = None
        self.unit_shard_bytes = np.zeros(0, np.int64)
        if units is not None:
            self.units = np.ascontiguousarray(units, dtype=np.int32)
            n_units = int(self.units.max()) + 1 if self.units.size else 0
            self.unit_shard_bytes = np.zeros(max(1, n_units), np.int64)
            L.n_units = n_units
            L.param_unit = self.units.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
            L.unit_shard_bytes = self.unit_shard_bytes.ctypes.data_as(_P64)
        self._explicit = None
        if explicit_offsets is not None:
            self._explicit = np.ascontiguousarray(explicit_offsets, dtype=np.int64)
            L.explicit_offset = self._explicit.ctypes.data_as(_P64)
        _check(lib().orc_layout_compute(ctypes.byref(L)), "layout")
        self.c = L
        self.param_offset = self.param_offset[:len(self.params)]
        self.chunk_rows = self.chunk_rows[:len(self.params)]
        self.param_gen_base = self.param_gen_base[:len(self.params)]
        self.tensor_numel = self.tensor_numel[:len(self.tensors)]
        self.tensor_offset = self.tensor_offset[:len(self.tensors)]
        self.flat_bytes = int(L.flat_bytes)
        self.shard_bytes = int(L.shard_bytes)
        self.n_buckets = int(self.rank_first_bucket[tp])
        if units is not None:
            self.unit_shard_bytes = self.unit_shard_bytes[:L.n_units]

    # -- source ---------------------------------------------------------------
    def param_numel(self, p: int) -> int:
        rows, cols = self.views[p]
        return rows * cols

    def host_shards(self, seed: int, specials: bool = False) -> List[np.ndarray]:
        """Materialise the source with the seeded generator and cut it into shards."""
        import synth
        if self.sharding == "tensors":
            out = []
            for p, (_, _, es) in enumerate(self.params):
                n = self.param_numel(p)
                vals = synth.values_host(n, es, seed, first_idx=int(self.param_gen_base[p]),
                                         specials=specials)
                out.append(vals.view(np.uint8).copy())
            return out
        if self.sharding == "units":
            # Each unit: its own flat buffer, cut into n_shards shards.
            out = []
            for u, Su in enumerate(self.unit_shard_bytes):
                Su = int(Su)
                flat = np.zeros(Su * self.n_shards, np.uint8)
                for p, (_, _, es) in enumerate(self.params):
                    if int(self.units[p]) != u:
                        continue
                    n = self.param_numel(p)
                    vals = synth.values_host(n, es, seed, first_idx=int(self.param_gen_base[p]),
                                             specials=specials)
                    off = int(self.param_offset[p])
                    flat[off:off + n * es] = vals.view(np.uint8)
                out += [flat[s * Su:(s + 1) * Su] for s in range(self.n_shards)]
            return out
        flat = np.zeros(self.shard_bytes * self.n_shards, np.uint8)
        S = self.shard_bytes
        for p, (_, _, es) in enumerate(self.params):
            rows, cols = self.views[p]
            base = int(self.param_gen_base[p])
            off = int(self.param_offset[p])
            if self.sharding == "flat":
                n = rows * cols
                vals = synth.values_host(n, es, seed, first_idx=base, specials=specials)
                flat[off:off + n * es] = vals.view(np.uint8)
                continue
            c = int(self.chunk_rows[p])
            for s in range(self.n_shards):
                r0, r1 = s * c, min((s + 1) * c, rows)
                if r1 <= r0:
                    continue
                n = (r1 - r0) * cols
                vals = synth.values_host(n, es, seed, first_idx=base + r0 * cols,
                                         specials=specials)
                flat[s * S + off:s * S + off + n * es] = vals.view(np.uint8)
        return [flat[s * S:(s + 1) * S] for s in range(self.n_shards)]

    # -- reshard / pack -------------------------------------------------------
    def reshard_tensor(self, src: Source, t: int) -> np.ndarray:
        out = np.empty(int(self.tensor_numel[t]), np.uint16)
        _check(lib().orc_reshard_tensor(ctypes.byref(self.c), ctypes.byref(src.c), t,
                                        out.ctypes.data), "reshard")
        return out

    def tensor_elements(self, src: Source, t: int, j0: int, j1: int) -> np.ndarray:
        out = np.empty(j1 - j0, np.uint16)
        _check(lib().orc_tensor_elements(ctypes.byref(self.c), ctypes.byref(src.c), t, j0, j1,
                                         out.ctypes.data), "tensor_elements")
        return out

    def pack_bucket(self, src: Source, b: int) -> np.ndarray:
        out = np.empty(self.bucket_bytes, np.uint8)
        _check(lib().orc_pack_bucket(ctypes.byref(self.c), ctypes.byref(src.c), b,
                                     out.ctypes.data), "pack_bucket")
        return out

    def pack(self, src: Source, first: int = 0, count: Optional[int] = None):
        """Buckets [first, first+count) as a [count, bucket_bytes] uint8 array, and checksums."""
        if count is None:
            count = self.n_buckets - first
        out = np.empty((count, self.bucket_bytes), np.uint8)
        cs = np.empty(count, np.uint64)
        _check(lib().orc_pack_range(ctypes.byref(self.c), ctypes.byref(src.c), first, count,
                                    out.ctypes.data, cs.ctypes.data), "pack_range")
        return out, cs

    # -- unpack / verify ------------------------------------------------------
    def _bucket_ptrs(self, buckets):
        ptrs = (ctypes.c_void_p * max(1, self.n_buckets))()
        keep = []
        if isinstance(buckets, np.ndarray) and buckets.ndim == 2:
            rows = [buckets[i] for i in range(buckets.shape[0])]
        else:
            rows = list(buckets)
        for i, b in enumerate(rows):
            if b is None:
                ptrs[i] = 0
                continue
            a = np.ascontiguousarray(b).view(np.uint8)
            assert a.size == self.bucket_bytes
            keep.append(a)
            ptrs[i] = a.ctypes.data
        return ptrs, keep

    def unpack_tensor(self, buckets, t: int) -> np.ndarray:
        ptrs, keep = self._bucket_ptrs(buckets)
        out = np.empty(int(self.tensor_numel[t]), np.uint16)
        _check(lib().orc_unpack_tensor(ctypes.byref(self.c), ptrs, t, out.ctypes.data),
               "unpack_tensor")
        del keep
        return out

    def unpack_elements(self, buckets, t: int, j0: int, j1: int) -> np.ndarray:
        ptrs, keep = self._bucket_ptrs(buckets)
        out = np.empty(j1 - j0, np.uint16)
        _check(lib().orc_unpack_elements(ctypes.byref(self.c), ptrs, t, j0, j1, out.ctypes.data),
               "unpack_elements")
        del keep
        return out

    def sync_sample(self, src: "Source", first: int, count: int) -> int:
        """One CPU weight sync restricted to buckets [first, first+count): pack
        them, unpack every tensor element that lies in them, verify them.
        Returns the algorithmic bytes of that sync, counted as for the GPU path:
        pack reads the source elements and writes the buckets; the receiver reads
        each bucket byte once (unpack and verify) and writes each element's two
        bytes."""
        packed, cs = self.pack(src, first, count)
        buckets = [None] * self.n_buckets
        for i in range(count):
            buckets[first + i] = packed[i]
        moved = 0
        for t, (_, rank, blocks) in enumerate(self.tensors):
            fb = int(self.rank_first_bucket[rank])
            lo = (first - fb) * self.bucket_bytes
            hi = (first + count - fb) * self.bucket_bytes
            t_lo = int(self.tensor_offset[t])
            t_hi = t_lo + 2 * int(self.tensor_numel[t])
            a, z = max(lo, t_lo), min(hi, t_hi)
            if a < z:
                self.unpack_elements(buckets, t, (a - t_lo) // 2, (z - t_lo) // 2)
                es = self.params[blocks[0][0]][2]
                moved += (z - a) // 2 * es      # pack: source bytes read
                moved += z - a                   # unpack: tensor bytes written
        full_cs = np.zeros(self.n_buckets, np.uint64)
        full_cs[first:first + count] = cs
        n_bad, _ = self.verify(buckets, full_cs, first, count)
        if n_bad:
            raise RuntimeError("oracle verify failed on its own buckets")
        moved += 2 * count * self.bucket_bytes   # pack writes, receiver reads
        return moved

    def verify(self, buckets, checksums, first: int = 0, count: Optional[int] = None):
        """(number of bad buckets, first bad index or -1)."""
        if count is None:
            count = self.n_buckets - first
        ptrs, keep = self._bucket_ptrs(buckets)
        cs = np.ascontiguousarray(checksums, dtype=np.uint64)
        fb = ctypes.c_int64(-1)
        n = lib().orc_verify(ctypes.byref(self.c), ptrs, cs.ctypes.data, first, count,
                             ctypes.byref(fb))
        del keep
        return int(n), int(fb.value)

    def tensor_index(self, name: str, rank: int = 0) -> int:
        for i, (n, r, _) in enumerate(self.tensors):
            if n == name and r == rank:
                return i
        raise KeyError((name, rank))


def workload_layout(w, bucket_bytes: Optional[int] = None) -> Layout:
    """Oracle layout for a ``synth.Workload``."""
    params = qwen3.manifest(w.shape, w.src_elem_bytes)
    tensors = qwen3.rollout_tensors(w.shape, params, w.tp, ep=getattr(w, "ep", False))
    units = qwen3.layer_units(params) if w.sharding == "units" else None
    return Layout(params, tensors, n_shards=w.n_shards, tp=w.tp,
                  bucket_bytes=bucket_bytes or w.bucket_bytes, sharding=w.sharding, units=units,
                  dst_dtype=getattr(w, "dst_dtype", "bf16"))
