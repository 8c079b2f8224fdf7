"""Python binding of the weight-sync C ABI (include/rr.h): argument marshalling only.

Every step of the path runs in the CUDA library ``librr.so``; this module
turns Python descriptions and torch tensors into the plain structs, pointers
and sizes that the ABI takes.  There is no fallback: if the library cannot be
loaded, importing this module raises.

Functions carry the ABI's names: ``rr_plan_create``, ``rr_pack``,
``rr_unpack``, ``rr_verify`` (RobustRL Section 5.2.1 steps 1-2 and
Section 5.2.2), plus the plan queries.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import List, Optional, Sequence

from . import build as _build

# ---------------------------------------------------------------------------
# Library
# ---------------------------------------------------------------------------

if not os.path.exists(_build.LIB):
    raise ImportError(
        f"{_build.LIB} is missing: build it with `python paper_2512_22492_gb300/build.py` "
        "(needs nvcc); there is no CPU fallback")
_lib = ctypes.CDLL(_build.LIB)

RR_OK, RR_EINVAL, RR_ENOMEM, RR_ECUDA, RR_ELAYOUT, RR_EMISMATCH = range(6)
RR_F32, RR_BF16 = 0, 1
(RR_ITEM_F32_VEC, RR_ITEM_F32_SCALAR, RR_ITEM_BF16_VEC, RR_ITEM_BF16_SCALAR, RR_ITEM_ZERO_VEC,
 RR_ITEM_ZERO_SCALAR, RR_ITEM_COPY_VEC, RR_ITEM_COPY_SCALAR) = range(8)


class _Param(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("ndim", ctypes.c_int32),
                ("shape", ctypes.c_int64 * 4), ("dtype", ctypes.c_int)]


class _SrcLayout(ctypes.Structure):
    _fields_ = [("n_shards", ctypes.c_int32), ("align_bytes", ctypes.c_int64),
                ("param_flat_offset", ctypes.POINTER(ctypes.c_int64)),
                ("sharding", ctypes.c_int32), ("shard_bytes", ctypes.c_int64),
                ("n_units", ctypes.c_int32), ("param_unit", ctypes.POINTER(ctypes.c_int32))]


class _Block(ctypes.Structure):
    _fields_ = [("param", ctypes.c_int32), ("row0", ctypes.c_int64), ("nrows", ctypes.c_int64),
                ("col0", ctypes.c_int64), ("ncols", ctypes.c_int64)]


class _DstTensor(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("rank", ctypes.c_int32), ("numel", ctypes.c_int64),
                ("n_blocks", ctypes.c_int32), ("blocks", ctypes.POINTER(_Block))]


class _DstLayout(ctypes.Structure):
    _fields_ = [("tp", ctypes.c_int32), ("n_tensors", ctypes.c_int32),
                ("tensors", ctypes.POINTER(_DstTensor)), ("tensor_align_bytes", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("reserved", ctypes.c_int32)]


_DST_DTYPES = {"bf16": 0, "f16": 1}


class _Options(ctypes.Structure):
    _fields_ = [("host_only", ctypes.c_int32), ("grid_blocks", ctypes.c_int32),
                ("chunk_bytes", ctypes.c_int64), ("engine", ctypes.c_int32),
                ("check_items", ctypes.c_int32)]


class _Stats(ctypes.Structure):
    _fields_ = [("n_pack_items", ctypes.c_int64), ("n_unpack_items", ctypes.c_int64),
                ("grid_blocks", ctypes.c_int32), ("unpack_grid_blocks", ctypes.c_int32),
                ("verify_grid_blocks", ctypes.c_int32), ("n_buckets", ctypes.c_int32),
                ("n_shards", ctypes.c_int32), ("n_tensors", ctypes.c_int32),
                ("bucket_bytes", ctypes.c_int64),
                ("pack_bytes_read", ctypes.c_int64), ("pack_bytes_written", ctypes.c_int64),
                ("unpack_bytes_read", ctypes.c_int64), ("unpack_bytes_written", ctypes.c_int64),
                ("verify_bytes_read", ctypes.c_int64), ("n_pack_full_items", ctypes.c_int64)]


class PackItem(ctypes.Structure):
    _fields_ = [("src", ctypes.c_uint64), ("dst_off", ctypes.c_uint32),
                ("bucket", ctypes.c_uint32), ("row_len", ctypes.c_uint32),
                ("n_rows", ctypes.c_uint32), ("src_stride", ctypes.c_uint32),
                ("kind", ctypes.c_uint16), ("reserved", ctypes.c_uint16)]


class UnpackItem(ctypes.Structure):
    _fields_ = [("dst_off", ctypes.c_uint64), ("src_off", ctypes.c_uint32),
                ("bucket", ctypes.c_uint32), ("tensor", ctypes.c_uint32),
                ("nbytes", ctypes.c_uint32), ("kind", ctypes.c_uint32),
                ("reserved", ctypes.c_uint32)]


def _np_dtype(struct):
    import numpy as np
    m = {ctypes.c_uint64: "<u8", ctypes.c_uint32: "<u4", ctypes.c_uint16: "<u2"}
    return np.dtype({"names": [f for f, _ in struct._fields_],
                     "formats": [m[t] for _, t in struct._fields_],
                     "offsets": [getattr(struct, f).offset for f, _ in struct._fields_],
                     "itemsize": ctypes.sizeof(struct)})


PACK_ITEM_DTYPE = _np_dtype(PackItem)
UNPACK_ITEM_DTYPE = _np_dtype(UnpackItem)

_vp = ctypes.c_void_p
_P64 = ctypes.POINTER(ctypes.c_int64)
_P32 = ctypes.POINTER(ctypes.c_int32)


def _sig(name, args, res=ctypes.c_int):
    f = getattr(_lib, name)
    f.argtypes = args
    f.restype = res
    return f


_sig("rr_plan_create_ex", [ctypes.POINTER(_Param), ctypes.c_int32, ctypes.POINTER(_SrcLayout),
                           ctypes.POINTER(_DstLayout), ctypes.c_size_t, ctypes.POINTER(_Options),
                           ctypes.POINTER(_vp)])
_sig("rr_plan_create", [ctypes.POINTER(_Param), ctypes.c_int32, ctypes.POINTER(_SrcLayout),
                        ctypes.POINTER(_DstLayout), ctypes.c_size_t, ctypes.POINTER(_vp)])
_sig("rr_plan_destroy", [_vp], None)
_sig("rr_plan_query", [_vp, _P32, _P64, _P32])
_sig("rr_plan_source", [_vp, _P64, _P64, _P64])
_sig("rr_plan_source_buffers", [_vp, _P32, _P64])
_sig("rr_plan_tensors", [_vp, _P64, _P64])
_sig("rr_plan_get_stats", [_vp, ctypes.POINTER(_Stats)])
_sig("rr_plan_export_pack", [_vp, ctypes.POINTER(PackItem), ctypes.c_int64,
                             ctypes.POINTER(ctypes.c_uint32)])
_sig("rr_plan_export_pack_full", [_vp, ctypes.POINTER(PackItem), ctypes.c_int64,
                                  ctypes.POINTER(ctypes.c_uint32)])
_sig("rr_plan_export_unpack", [_vp, ctypes.POINTER(UnpackItem), ctypes.c_int64,
                               ctypes.POINTER(ctypes.c_uint32)])
_sig("rr_pack", [_vp, ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp, _vp])
_sig("rr_unpack", [_vp, ctypes.POINTER(_vp), ctypes.POINTER(_vp), _vp])
_sig("rr_verify", [_vp, ctypes.POINTER(_vp), _vp, _P64, _P64, _vp])
_sig("rr_pack_range", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp),
                       ctypes.POINTER(_vp), _vp, _vp])
_sig("rr_unpack_range", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp),
                         ctypes.POINTER(_vp), _vp])
_sig("rr_verify_range", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp), _vp, _vp, _P64,
                         _P64, _vp])
_sig("rr_unpack_verify", [_vp, ctypes.POINTER(_vp), _vp, ctypes.POINTER(_vp), _vp, _P64, _P64, _vp])
_sig("rr_unpack_verify_range", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp), _vp,
                                ctypes.POINTER(_vp), _vp, _P64, _P64, _vp])
_sig("rr_clear_range", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp), _vp])
_sig("rr_unpack_verify_async", [_vp, ctypes.c_int32, ctypes.c_int32, ctypes.POINTER(_vp), _vp,
                                ctypes.POINTER(_vp), _vp, _vp, _vp, _vp])
_sig("rr_plan_bucket_items", [_vp, ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_uint32)])
_sig("rr_plan_work_units", [_vp, ctypes.c_int32, ctypes.POINTER(ctypes.c_int32),
                            ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_uint32)])
_sig("rr_verify_noalloc", [ctypes.POINTER(_vp), ctypes.c_int32, ctypes.c_size_t, _vp, _P64, _P64,
                           _vp])
_sig("rr_plan_check", [_vp, _vp])
_sig("rr_plan_selftest_wait", [_vp, _vp])
_sig("rr_status_str", [ctypes.c_int], ctypes.c_char_p)
_sig("rr_last_error", [], ctypes.c_char_p)

LIBRARY_PATH = _build.LIB
EXPORTED = ("rr_plan_create", "rr_plan_create_ex", "rr_plan_destroy", "rr_plan_query",
            "rr_plan_source", "rr_plan_source_buffers", "rr_plan_tensors", "rr_plan_get_stats",
            "rr_plan_export_pack", "rr_plan_export_pack_full",
            "rr_plan_export_unpack", "rr_plan_bucket_items", "rr_plan_work_units", "rr_pack", "rr_unpack", "rr_verify",
            "rr_pack_range", "rr_unpack_range", "rr_verify_range", "rr_clear_range",
            "rr_unpack_verify", "rr_unpack_verify_range", "rr_unpack_verify_async",
            "rr_verify_noalloc",
            "rr_plan_check", "rr_plan_selftest_wait", "rr_status_str", "rr_last_error")


class RRError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        detail = _lib.rr_last_error().decode()
        super().__init__(f"{what}: {_lib.rr_status_str(status).decode()}"
                         + (f" ({detail})" if detail else ""))


def _check(status: int, what: str) -> None:
    if status != RR_OK:
        raise RRError(status, what)


def rr_status_str(status: int) -> str:
    return _lib.rr_status_str(status).decode()


# ---------------------------------------------------------------------------
# Descriptions
# ---------------------------------------------------------------------------

@dataclass
class Param:
    name: str
    shape: Sequence[int]
    dtype: str = "f32"    # "f32" or "bf16"


@dataclass
class SrcLayout:
    n_shards: int
    align_bytes: int = 16
    param_flat_offset: Optional[Sequence[int]] = None
    sharding: str = "flat"    # "flat" (FSDP1 FlatParameter), "rows" (FSDP2 dim-0 Shard),
                              # "tensors" (one buffer per parameter), or "units" (FSDP1,
                              # one FlatParameter per wrapped module)
    shard_bytes: int = 0      # flat only: explicit shard size, 0 = computed
    units: Optional[Sequence[int]] = None   # units only: the unit of each parameter


@dataclass
class Block:
    param: int
    row0: int
    nrows: int
    col0: int
    ncols: int


@dataclass
class DstTensor:
    name: str
    rank: int
    blocks: List[Block]
    numel: Optional[int] = None   # default: sum of the blocks

    def size(self) -> int:
        return sum(b.nrows * b.ncols for b in self.blocks) if self.numel is None else self.numel


@dataclass
class DstLayout:
    tp: int
    tensors: List[DstTensor]
    tensor_align_bytes: int = 256
    dtype: str = "bf16"      # the rollout's 16-bit element type: "bf16" or "f16"


@dataclass
class PlanOptions:
    host_only: bool = False
    grid_blocks: int = 0
    chunk_bytes: int = 0
    engine: str = "auto"      # "auto" (bulk-copy engine for device buffers) or "registers"
    check_items: bool = False  # kernels check every work item's bounds (a debugging aid)


# ---------------------------------------------------------------------------
# Plan
# ---------------------------------------------------------------------------

class Plan:
    """Owns an rr_plan; exposes its geometry."""

    def __init__(self, handle: int, n_params: int, dst: DstLayout, src: SrcLayout = None):
        self._h = ctypes.c_void_p(handle)
        self.n_params = n_params
        self.dst_dtype = dst.dtype
        self.sharding = src.sharding if src else "flat"
        self.align_bytes = src.align_bytes if src else 16
        self.tp = dst.tp
        self.n_tensors = len(dst.tensors)
        self.tensor_names = [t.name for t in dst.tensors]
        self.tensor_ranks = [t.rank for t in dst.tensors]
        st = self.stats()
        self.n_buckets = st["n_buckets"]
        self.bucket_bytes = st["bucket_bytes"]
        self.n_shards = st["n_shards"]
        self.grid_blocks = st["grid_blocks"]
        self._unpack_grid = st["unpack_grid_blocks"]
        sb = (ctypes.c_int64 * self.tp)()
        fb = (ctypes.c_int32 * (self.tp + 1))()
        nb = ctypes.c_int32()
        _check(_lib.rr_plan_query(self._h, ctypes.byref(nb), sb, fb), "rr_plan_query")
        self.stream_bytes_per_rank = list(sb)
        self.first_bucket_of_rank = list(fb)
        shard = ctypes.c_int64()
        flat = ctypes.c_int64()
        offs = (ctypes.c_int64 * max(1, n_params))()
        _check(_lib.rr_plan_source(self._h, ctypes.byref(shard), ctypes.byref(flat), offs),
               "rr_plan_source")
        self.shard_bytes = shard.value
        self.flat_bytes = flat.value
        self.param_flat_offset = list(offs)[:n_params]
        nbuf = ctypes.c_int32()
        _check(_lib.rr_plan_source_buffers(self._h, ctypes.byref(nbuf), None),
               "rr_plan_source_buffers")
        sizes = (ctypes.c_int64 * max(1, nbuf.value))()
        _check(_lib.rr_plan_source_buffers(self._h, None, sizes), "rr_plan_source_buffers")
        self.source_buffer_bytes = list(sizes)[:nbuf.value]
        self.units = list(src.units) if src is not None and src.units is not None else None
        numel = (ctypes.c_int64 * max(1, self.n_tensors))()
        toff = (ctypes.c_int64 * max(1, self.n_tensors))()
        _check(_lib.rr_plan_tensors(self._h, numel, toff), "rr_plan_tensors")
        self.tensor_numel = list(numel)[:self.n_tensors]
        self.tensor_stream_offset = list(toff)[:self.n_tensors]

    @property
    def handle(self) -> ctypes.c_void_p:
        if not self._h:
            raise ValueError("plan destroyed")
        return self._h

    def stats(self) -> dict:
        s = _Stats()
        _check(_lib.rr_plan_get_stats(self._h, ctypes.byref(s)), "rr_plan_get_stats")
        return {k: getattr(s, k) for k, _ in _Stats._fields_}

    def export_pack(self):
        """(items as a numpy structured array, per-block first item)."""
        import numpy as np
        n = self.stats()["n_pack_items"]
        items = np.zeros(max(1, n), dtype=PACK_ITEM_DTYPE)
        first = np.zeros(self.stats()["grid_blocks"] + 1, dtype=np.uint32)
        _check(_lib.rr_plan_export_pack(self._h, items.ctypes.data_as(ctypes.POINTER(PackItem)),
                                        n, first.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32))),
               "rr_plan_export_pack")
        return items[:n], first

    def export_pack_full(self):
        """The whole-sync pack table (fan-out groups included) and its per-block
        first item, as rr_pack runs it on the bulk-copy engine for every bucket."""
        import numpy as np
        n = self.stats()["n_pack_full_items"]
        items = np.zeros(max(1, n), dtype=PACK_ITEM_DTYPE)
        first = np.zeros(self.stats()["grid_blocks"] + 1, dtype=np.uint32)
        _check(_lib.rr_plan_export_pack_full(
            self._h, items.ctypes.data_as(ctypes.POINTER(PackItem)), n,
            first.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32))), "rr_plan_export_pack_full")
        return items[:n], first

    def export_unpack(self):
        import numpy as np
        n = self.stats()["n_unpack_items"]
        items = np.zeros(max(1, n), dtype=UNPACK_ITEM_DTYPE)
        # The unpack table is cut for the unpack kernel's own grid.
        first = np.zeros(self._unpack_grid + 1, dtype=np.uint32)
        _check(_lib.rr_plan_export_unpack(self._h,
                                          items.ctypes.data_as(ctypes.POINTER(UnpackItem)), n,
                                          first.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32))),
               "rr_plan_export_unpack")
        return items[:n], first

    def bucket_items(self):
        """Per-bucket first item of the pack and unpack tables (n_buckets + 1 each)."""
        import numpy as np
        pf = np.zeros(self.n_buckets + 1, np.uint32)
        uf = np.zeros(self.n_buckets + 1, np.uint32)
        P = ctypes.POINTER(ctypes.c_uint32)
        _check(_lib.rr_plan_bucket_items(self._h, pf.ctypes.data_as(P), uf.ctypes.data_as(P)),
               "rr_plan_bucket_items")
        return pf, uf

    def work_units(self, which: str = "unpack"):
        """The bulk-copy engine's work units: "pack" and "unpack" (per bucket:
        bucket-range packs, every unpack) or "pack_full" (a pack over every
        bucket).  Returns (first item of each unit, plus one past the last;
        first unit of each bucket, n_buckets + 1, or None for "pack_full")."""
        import numpy as np
        w = {"pack": 0, "pack_full": 1, "unpack": 2}[which]
        n = ctypes.c_int32(0)
        _check(_lib.rr_plan_work_units(self._h, w, ctypes.byref(n), None, None),
               "rr_plan_work_units")
        first = np.zeros(n.value + 1, np.uint32)
        bucket = None if which.endswith("_full") else np.zeros(self.n_buckets + 1, np.uint32)
        P = ctypes.POINTER(ctypes.c_uint32)
        _check(_lib.rr_plan_work_units(self._h, w, ctypes.byref(n), first.ctypes.data_as(P),
                                       None if bucket is None else bucket.ctypes.data_as(P)),
               "rr_plan_work_units")
        return first, bucket

    def destroy(self) -> None:
        if self._h:
            _lib.rr_plan_destroy(self._h)
            self._h = ctypes.c_void_p(0)

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def rr_plan_create(manifest: Sequence[Param], src: SrcLayout, dst: DstLayout,
                   bucket_bytes: int, options: Optional[PlanOptions] = None) -> Plan:
    n = len(manifest)
    cp = (_Param * max(1, n))()
    names = []
    for i, p in enumerate(manifest):
        nm = p.name.encode()
        names.append(nm)
        cp[i].name = nm
        cp[i].ndim = len(p.shape)
        for d, s in enumerate(p.shape):
            cp[i].shape[d] = s
        cp[i].dtype = RR_F32 if p.dtype == "f32" else RR_BF16
    cs = _SrcLayout(n_shards=src.n_shards, align_bytes=src.align_bytes,
                    sharding={"flat": 0, "rows": 1, "tensors": 2, "units": 3}[src.sharding],
                    shard_bytes=src.shard_bytes)
    offs = None
    if src.param_flat_offset is not None:
        offs = (ctypes.c_int64 * max(1, n))(*src.param_flat_offset)
        cs.param_flat_offset = offs
    units = None
    if src.units is not None:
        units = (ctypes.c_int32 * max(1, len(src.units)))(*src.units)
        cs.n_units = max(src.units) + 1 if len(src.units) else 0
        cs.param_unit = units
    keep = []
    ct = (_DstTensor * max(1, len(dst.tensors)))()
    for i, t in enumerate(dst.tensors):
        cb = (_Block * max(1, len(t.blocks)))()
        for k, b in enumerate(t.blocks):
            cb[k].param, cb[k].row0, cb[k].nrows, cb[k].col0, cb[k].ncols = \
                b.param, b.row0, b.nrows, b.col0, b.ncols
        nm = t.name.encode()
        keep += [cb, nm]
        ct[i].name = nm
        ct[i].rank = t.rank
        ct[i].numel = t.size()
        ct[i].n_blocks = len(t.blocks)
        ct[i].blocks = ctypes.cast(cb, ctypes.POINTER(_Block))
    if dst.dtype not in _DST_DTYPES:
        raise ValueError(f"destination dtype must be one of {sorted(_DST_DTYPES)}, "
                         f"not {dst.dtype!r}")
    cd = _DstLayout(tp=dst.tp, n_tensors=len(dst.tensors),
                    tensors=ctypes.cast(ct, ctypes.POINTER(_DstTensor)),
                    tensor_align_bytes=dst.tensor_align_bytes, dtype=_DST_DTYPES[dst.dtype])
    out = ctypes.c_void_p()
    if options is None:
        st = _lib.rr_plan_create(cp, n, ctypes.byref(cs), ctypes.byref(cd), bucket_bytes,
                                 ctypes.byref(out))
    else:
        co = _Options(host_only=int(options.host_only), grid_blocks=options.grid_blocks,
                      chunk_bytes=options.chunk_bytes,
                      engine={"auto": 0, "registers": 1}[options.engine],
                      check_items=int(options.check_items))
        st = _lib.rr_plan_create_ex(cp, n, ctypes.byref(cs), ctypes.byref(cd), bucket_bytes,
                                    ctypes.byref(co), ctypes.byref(out))
    _check(st, "rr_plan_create")
    plan = Plan(out.value, n, dst, src)
    plan.param_bytes = []
    for p in manifest:
        numel = 1
        for d in p.shape:
            numel *= d
        plan.param_bytes.append(numel * (4 if p.dtype == "f32" else 2))
    return plan


# ---------------------------------------------------------------------------
# Pointers and streams
# ---------------------------------------------------------------------------

def _ptr(x) -> int:
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _ptr_array(xs) -> ctypes.Array:
    """Host array of device pointers from tensors / ints, or the rows of a 2-D tensor."""
    if isinstance(xs, Pointers):
        return xs.array
    if hasattr(xs, "dim") and xs.dim() == 2:
        base = xs.data_ptr()
        step = xs.stride(0) * xs.element_size()
        ptrs = [base + i * step for i in range(xs.shape[0])]
    else:
        ptrs = [_ptr(x) for x in xs]
    return (ctypes.c_void_p * max(1, len(ptrs)))(*ptrs)


def _stream(stream) -> int:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


# ---------------------------------------------------------------------------
# Hot path
# ---------------------------------------------------------------------------

def _nbytes(x):
    """Byte size of a tensor argument, or None for a raw pointer (unchecked)."""
    if isinstance(x, int):
        return None
    return int(x.numel()) * int(x.element_size())


def _check_list(xs, n: int, min_bytes, what: str, plan: Optional[Plan] = None) -> None:
    """Host arrays handed to the ABI hold exactly n pointers; tensor arguments
    must be large enough for what the plan will write or read."""
    if isinstance(xs, Pointers):
        if xs.role != what:
            raise ValueError(f"{what}: pointer table was built for {xs.role}")
        if xs.n != n:
            raise ValueError(f"{what}: {xs.n} entries, plan expects {n}")
        if plan is not None and xs.plan is plan:
            return                      # validated against this plan when it was built
        for i, nb in enumerate(xs.sizes):
            need = min_bytes(i) if callable(min_bytes) else min_bytes
            if nb is not None and need is not None and nb < need:
                raise ValueError(f"{what}[{i}]: {nb} bytes, plan needs {need}")
        return
    if hasattr(xs, "dim") and xs.dim() == 2:
        if xs.shape[0] != n:
            raise ValueError(f"{what}: {xs.shape[0]} rows, plan expects {n}")
        if xs.shape[0] > 1 and (xs.stride(1) != 1 or xs.stride(0) < xs.shape[1]):
            raise ValueError(f"{what}: rows must be contiguous and must not overlap")
        if min_bytes is not None and xs.shape[1] * xs.element_size() < min_bytes:
            raise ValueError(f"{what}: rows of {xs.shape[1] * xs.element_size()} bytes, plan "
                             f"needs {min_bytes}")
        return
    xs = list(xs)
    if len(xs) != n:
        raise ValueError(f"{what}: {len(xs)} entries, plan expects {n}")
    for i, x in enumerate(xs):
        if hasattr(x, "is_contiguous") and not x.is_contiguous():
            raise ValueError(f"{what}[{i}]: not contiguous (the library writes and reads its "
                             f"bytes in order)")
        need = min_bytes(i) if callable(min_bytes) else min_bytes
        nb = _nbytes(x)
        if nb is not None and need is not None and nb < need:
            raise ValueError(f"{what}[{i}]: {nb} bytes, plan needs {need}")


_ROLES = ("src_shards", "buckets", "dst")


def _role_need(plan: Plan, role: str):
    if role == "src_shards":
        return plan.n_shards, _shard_need(plan)
    if role == "buckets":
        return plan.n_buckets, plan.bucket_bytes
    return plan.n_tensors, lambda i: 2 * plan.tensor_numel[i]


class Pointers:
    """A pointer table checked against a plan and marshalled once.

    Pass it wherever a call takes `src_shards`, `buckets` or `dst` (the role it
    was built for).  A list of tensors is otherwise walked on every call --
    sizes checked, pointers gathered into a host array -- which for a rollout
    layout of a few thousand destination tensors costs about a millisecond of
    host time per call.  The table holds references to the tensors it was
    built from; they must not be resized or freed while it is in use."""

    def __init__(self, plan: Plan, role: str, xs):
        if role not in _ROLES:
            raise ValueError(f"role must be one of {_ROLES}, not {role!r}")
        n, need = _role_need(plan, role)
        _check_list(xs, n, need, role, plan=plan)
        self.plan = plan
        self.role = role
        self.n = n
        self.array = _ptr_array(xs)
        if hasattr(xs, "dim") and xs.dim() == 2:
            self.sizes = [int(xs.shape[1]) * int(xs.element_size())] * n
        else:
            self.sizes = [_nbytes(x) for x in xs]
        self._keep = xs

    def __len__(self) -> int:
        return self.n


def _check_checksums(plan: Plan, checksums) -> None:
    if hasattr(checksums, "is_contiguous") and not checksums.is_contiguous():
        raise ValueError("checksums: not contiguous")
    nb = _nbytes(checksums)
    if nb is not None and nb < 8 * plan.n_buckets:
        raise ValueError(f"checksums: {nb} bytes, plan needs {8 * plan.n_buckets}")


def _shard_need(plan: Plan):
    if plan.sharding in ("tensors", "units"):
        return lambda i: plan.source_buffer_bytes[i]
    return plan.shard_bytes


def rr_pack(plan: Plan, src_shards, buckets, checksums, stream=None) -> None:
    """Reshard + cast + pack + checksum (asynchronous on `stream`)."""
    _check_list(src_shards, plan.n_shards, _shard_need(plan), "src_shards", plan=plan)
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_checksums(plan, checksums)
    _check(_lib.rr_pack(plan.handle, _ptr_array(src_shards), _ptr_array(buckets),
                        _ptr(checksums), _stream(stream)), "rr_pack")


def rr_unpack(plan: Plan, buckets, dst, stream=None) -> None:
    """Buckets -> destination tensors (asynchronous on `stream`)."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_list(dst, plan.n_tensors, lambda i: 2 * plan.tensor_numel[i], "dst", plan=plan)
    _check(_lib.rr_unpack(plan.handle, _ptr_array(buckets), _ptr_array(dst), _stream(stream)),
           "rr_unpack")


def rr_verify(plan: Plan, buckets, checksums, stream=None):
    """Recompute and compare checksums; returns (n_bad, first_bad).  Synchronous."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_checksums(plan, checksums)
    n_bad = ctypes.c_int64()
    first = ctypes.c_int64()
    st = _lib.rr_verify(plan.handle, _ptr_array(buckets), _ptr(checksums), ctypes.byref(n_bad),
                        ctypes.byref(first), _stream(stream))
    if st not in (RR_OK, RR_EMISMATCH):
        _check(st, "rr_verify")
    return n_bad.value, first.value


def rr_pack_range(plan: Plan, first_bucket: int, n_buckets: int, src_shards, buckets, checksums,
                  stream=None) -> None:
    """Pack only buckets [first_bucket, first_bucket + n_buckets) (asynchronous)."""
    _check_list(src_shards, plan.n_shards, _shard_need(plan), "src_shards", plan=plan)
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_checksums(plan, checksums)
    _check(_lib.rr_pack_range(plan.handle, first_bucket, n_buckets, _ptr_array(src_shards),
                              _ptr_array(buckets), _ptr(checksums), _stream(stream)),
           "rr_pack_range")


def rr_unpack_range(plan: Plan, first_bucket: int, n_buckets: int, buckets, dst,
                    stream=None) -> None:
    """Unpack only the destination bytes held by those buckets (asynchronous)."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_list(dst, plan.n_tensors, lambda i: 2 * plan.tensor_numel[i], "dst", plan=plan)
    _check(_lib.rr_unpack_range(plan.handle, first_bucket, n_buckets, _ptr_array(buckets),
                                _ptr_array(dst), _stream(stream)), "rr_unpack_range")


def rr_verify_range(plan: Plan, first_bucket: int, n_buckets: int, buckets, checksums, bad=None,
                    stream=None):
    """Verify those buckets; optional device byte array `bad` gets one flag per
    bucket of the range.  Returns (n_bad, first_bad).  Synchronous."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_checksums(plan, checksums)
    if bad is not None and _nbytes(bad) is not None and _nbytes(bad) < n_buckets:
        raise ValueError(f"bad: {_nbytes(bad)} bytes, need {n_buckets}")
    n_bad = ctypes.c_int64()
    first = ctypes.c_int64()
    st = _lib.rr_verify_range(plan.handle, first_bucket, n_buckets, _ptr_array(buckets),
                              _ptr(checksums), None if bad is None else _ptr(bad),
                              ctypes.byref(n_bad), ctypes.byref(first), _stream(stream))
    if st not in (RR_OK, RR_EMISMATCH):
        _check(st, "rr_verify_range")
    return n_bad.value, first.value


def rr_unpack_verify(plan: Plan, buckets, checksums, dst, bad=None, stream=None,
                     first_bucket: int = 0, n_buckets: Optional[int] = None):
    """Unpack and verify in one pass over the buckets (optionally a bucket range).
    Returns (n_bad, first_bad).  Synchronous."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_list(dst, plan.n_tensors, lambda i: 2 * plan.tensor_numel[i], "dst", plan=plan)
    _check_checksums(plan, checksums)
    n = plan.n_buckets - first_bucket if n_buckets is None else n_buckets
    if bad is not None and _nbytes(bad) is not None and _nbytes(bad) < n:
        raise ValueError(f"bad: {_nbytes(bad)} bytes, need {n}")
    n_bad = ctypes.c_int64()
    first = ctypes.c_int64()
    badp = None if bad is None else _ptr(bad)
    if first_bucket == 0 and n_buckets is None:
        st = _lib.rr_unpack_verify(plan.handle, _ptr_array(buckets), _ptr(checksums),
                                   _ptr_array(dst), badp, ctypes.byref(n_bad), ctypes.byref(first),
                                   _stream(stream))
    else:
        st = _lib.rr_unpack_verify_range(plan.handle, first_bucket, n, _ptr_array(buckets),
                                         _ptr(checksums), _ptr_array(dst), badp,
                                         ctypes.byref(n_bad), ctypes.byref(first), _stream(stream))
    if st not in (RR_OK, RR_EMISMATCH):
        _check(st, "rr_unpack_verify")
    return n_bad.value, first.value


def rr_unpack_verify_async(plan: Plan, buckets, checksums, dst, scratch, result, bad=None,
                           stream=None, first_bucket: int = 0,
                           n_buckets: Optional[int] = None) -> None:
    """Stream-ordered unpack + verify: returns after enqueueing.  `scratch` is a
    device tensor of at least n_buckets + 4 int64 (reused only after `result`
    is written); `result` (2 int64, device or pinned host memory) receives
    {n_bad, first_bad or -1} when the work on `stream` is done."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check_list(dst, plan.n_tensors, lambda i: 2 * plan.tensor_numel[i], "dst", plan=plan)
    _check_checksums(plan, checksums)
    n = plan.n_buckets - first_bucket if n_buckets is None else n_buckets
    for what, x, need in (("scratch", scratch, 8 * (n + 4)), ("result", result, 16),
                          ("bad", bad, n)):
        if x is not None and _nbytes(x) is not None and _nbytes(x) < need:
            raise ValueError(f"{what}: {_nbytes(x)} bytes, need {need}")
    _check(_lib.rr_unpack_verify_async(plan.handle, first_bucket, n, _ptr_array(buckets),
                                       _ptr(checksums), _ptr_array(dst),
                                       None if bad is None else _ptr(bad), _ptr(scratch),
                                       _ptr(result), _stream(stream)), "rr_unpack_verify_async")


def rr_clear_range(plan: Plan, first_bucket: int, n_buckets: int, buckets, stream=None) -> None:
    """Zero-fill buckets [first_bucket, first_bucket + n_buckets) (asynchronous)."""
    _check_list(buckets, plan.n_buckets, plan.bucket_bytes, "buckets", plan=plan)
    _check(_lib.rr_clear_range(plan.handle, first_bucket, n_buckets, _ptr_array(buckets),
                               _stream(stream)), "rr_clear_range")


def rr_plan_check(plan: Plan, stream=None) -> None:
    """Raise if a kernel of this plan gave up on a bounded wait (waits for `stream`)."""
    _check(_lib.rr_plan_check(plan.handle, _stream(stream)), "rr_plan_check")


def rr_plan_selftest_wait(plan: Plan, stream=None) -> None:
    """Enqueue the bounded-wait self-test kernel (see include/rr.h)."""
    _check(_lib.rr_plan_selftest_wait(plan.handle, _stream(stream)), "rr_plan_selftest_wait")


def rr_verify_noalloc(buckets, n_buckets: int, bucket_bytes: int, checksums, stream=None):
    """Allocation-free checksum check, for callers that cannot allocate device
    memory at that moment (e.g. an inference engine that has reserved almost all
    of it).  No plan needed; returns (n_bad, first_bad).  Synchronous; at most
    16384 buckets; overlapping calls share one device scratch array and race."""
    _check_list(buckets, n_buckets, bucket_bytes, "buckets")
    nb = _nbytes(checksums)
    if nb is not None and nb < 8 * n_buckets:
        raise ValueError(f"checksums: {nb} bytes, need {8 * n_buckets}")
    n_bad = ctypes.c_int64()
    first = ctypes.c_int64()
    st = _lib.rr_verify_noalloc(_ptr_array(buckets), n_buckets, bucket_bytes, _ptr(checksums),
                                ctypes.byref(n_bad), ctypes.byref(first), _stream(stream))
    if st not in (RR_OK, RR_EMISMATCH):
        _check(st, "rr_verify_noalloc")
    return n_bad.value, first.value
