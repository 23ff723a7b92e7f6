"""Thin ctypes binding of libwt.so (include/wt.h), same names as the C ABI.

Argument marshalling only: every step of the path runs in the library's C++
and CUDA code.  Pointers are plain integers (``tensor.data_ptr()``), streams
are ``torch.cuda.Stream.cuda_stream`` integers; PyTorch supplies device memory
and streams and nothing else.  There is no fallback: if the library cannot be
loaded, every call raises.
"""
from __future__ import annotations

import ctypes as C
import os
from dataclasses import dataclass
from typing import List, Sequence, Tuple

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libwt.so")

WT_OK, WT_EINVAL, WT_EIO, WT_EFORMAT, WT_ENOMEM, WT_ECUDA, WT_ENOTSUP, WT_ETIMEDOUT = 0, -1, -2, -3, -4, -5, -6, -7
WT_F32, WT_BF16, WT_F16, WT_I8, WT_U8 = 0, 1, 2, 3, 4
WT_ROUTE_AUTO, WT_ROUTE_REGISTER, WT_ROUTE_DIRECT, WT_ROUTE_NONE = 0, 1, 2, 3
WT_OPEN_HOST_ONLY, WT_OPEN_PREFAULT, WT_OPEN_TIMELINE, WT_OPEN_NOMAP = 1 << 4, 1 << 5, 1 << 6, 1 << 7
WT_OPEN_STAMPS, WT_OPEN_MAP_LARGE = 1 << 8, 1 << 9
WT_MAP_MIN_BYTES = 1 << 18
# the per-CTA record of wt_pass_stamps, in field order
STAMP_FIELDS = ("entry", "prologue", "operands", "first_copy", "first_full", "last_full", "exit", "sm")
WT_TRACE_INGEST, WT_TRACE_GEMV = 0, 1
WT_ADOPT_GATHER, WT_ADOPT_CE, WT_ADOPT_STAGED = 0, 1, 2
ROUTE_NAMES = {WT_ROUTE_REGISTER: "register", WT_ROUTE_DIRECT: "direct", WT_ROUTE_NONE: "none"}
MODE_NAMES = {WT_ADOPT_GATHER: "gather", WT_ADOPT_CE: "ce", WT_ADOPT_STAGED: "staged"}

# every entry point declared in include/wt.h
SYMBOLS = ("wt_last_error", "wt_abi_version", "wt_open", "wt_num_tensors", "wt_num_files",
           "wt_tensor_info", "wt_tensor_table", "wt_tensor_names", "wt_tensor_groups", "wt_find",
           "wt_file_route", "wt_file_registration", "wt_adopt", "wt_pass", "wt_checksum",
           "wt_checksum_plain", "wt_checksum_noalloc", "wt_device_status", "wt_residency",
           "wt_kernel_launches", "wt_trace", "wt_pass_stamps", "wt_open_times", "wt_live", "wt_close",
           # include/wt_dlpack.h
           "wt_dlpack_file", "wt_dlpack_tensor", "wt_dlpack_release", "wt_dlpack_live")
WT_DLPACK_DEVICE, WT_DLPACK_HOST = 0, 1
kDLCPU, kDLCUDA = 1, 2


class WtError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__("wt error %d: %s" % (code, msg))
        self.code = code


class TensorMeta(C.Structure):
    _fields_ = [("name", C.c_char_p), ("dtype", C.c_int32), ("ndim", C.c_int32),
                ("shape", C.c_uint64 * 4), ("nbytes", C.c_uint64), ("file", C.c_uint32),
                ("offset", C.c_uint64), ("host_ptr", C.c_void_p)]


class GemvDesc(C.Structure):
    _fields_ = [("W", C.c_void_p), ("dtype", C.c_int32), ("cols", C.c_int32),
                ("M", C.c_uint64), ("K", C.c_uint64), ("x", C.c_void_p), ("y", C.c_void_p),
                ("wait_event", C.c_void_p), ("scale", C.c_void_p)]


class LiveCounts(C.Structure):
    _fields_ = [("handles", C.c_int64), ("plans", C.c_int64), ("events", C.c_int64),
                ("device_bytes", C.c_int64), ("pinned_bytes", C.c_int64),
                ("cached_device_bytes", C.c_int64), ("cached_pinned_bytes", C.c_int64)]


class TraceRec(C.Structure):
    _fields_ = [("kind", C.c_int32), ("pad", C.c_int32), ("index", C.c_uint64), ("bytes", C.c_uint64),
                ("event", C.c_void_p), ("begin_ms", C.c_double), ("end_ms", C.c_double)]


# wt_tensor_meta as a numpy record (wt_tensor_table fills an array of them in one call).
META_DTYPE = np.dtype([("name", "<u8"), ("dtype", "<i4"), ("ndim", "<i4"), ("shape", "<u8", (4,)),
                       ("nbytes", "<u8"), ("file", "<u4"), ("pad", "<u4"), ("offset", "<u8"), ("host_ptr", "<u8")])
assert META_DTYPE.itemsize == C.sizeof(TensorMeta)


# The same 64-byte layout as a numpy record, for building many descriptors at once.
DESC_DTYPE = np.dtype([("W", "<u8"), ("dtype", "<i4"), ("cols", "<i4"), ("M", "<u8"), ("K", "<u8"),
                       ("x", "<u8"), ("y", "<u8"), ("wait_event", "<u8"), ("scale", "<u8")])
assert DESC_DTYPE.itemsize == C.sizeof(GemvDesc)


_lib = None
ABI_VERSION = 4  # wt_abi_version() of the include/wt.h this binding follows


def lib(path: str = LIB_PATH):
    """Load libwt.so (built by paper_2608_12114_gb300.build).  Raises if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError("libwt.so is not built (%s); run paper_2608_12114_gb300.build.build()" % path)
    L = C.CDLL(path)
    vp, sz, u64p = C.c_void_p, C.c_size_t, C.POINTER(C.c_uint64)
    L.wt_last_error.restype = C.c_char_p
    L.wt_abi_version.restype = C.c_int
    if L.wt_abi_version() != ABI_VERSION:  # a stale build: structures would not match
        raise RuntimeError("%s has ABI version %d, this binding needs %d; rebuild it"
                           % (path, L.wt_abi_version(), ABI_VERSION))
    L.wt_open.argtypes = [C.POINTER(C.c_char_p), C.c_int, C.c_uint, C.POINTER(vp)]
    L.wt_num_tensors.argtypes = [vp, C.POINTER(sz)]
    L.wt_num_files.argtypes = [vp, C.POINTER(sz)]
    L.wt_tensor_info.argtypes = [vp, sz, C.POINTER(TensorMeta)]
    L.wt_tensor_table.argtypes = [vp, sz, sz, vp]
    L.wt_tensor_names.argtypes = [vp, C.c_char_p, sz, C.POINTER(sz)]
    L.wt_tensor_groups.argtypes = [vp, vp, vp, C.POINTER(sz)]
    L.wt_find.argtypes = [vp, C.c_char_p, C.POINTER(sz)]
    L.wt_file_route.argtypes = [vp, sz, C.POINTER(C.c_uint)]
    L.wt_file_registration.argtypes = [vp, sz, C.POINTER(C.c_uint)]
    L.wt_adopt.argtypes = [vp, vp, vp, sz, C.c_uint, vp, vp]
    L.wt_pass.argtypes = [vp, C.POINTER(GemvDesc), sz, vp]
    L.wt_checksum.argtypes = [vp, C.POINTER(vp), u64p, sz, vp, vp]
    L.wt_checksum_plain.argtypes = [vp, C.POINTER(vp), u64p, sz, vp, vp]
    L.wt_checksum_noalloc.argtypes = [C.POINTER(vp), u64p, sz, vp, vp]
    L.wt_device_status.argtypes = [vp, C.POINTER(C.c_int)]
    L.wt_kernel_launches.argtypes = [vp, u64p]
    L.wt_residency.argtypes = [vp, u64p, u64p]
    L.wt_trace.argtypes = [vp, vp, C.POINTER(TraceRec), sz, C.POINTER(sz)]
    L.wt_pass_stamps.argtypes = [vp, vp, sz, C.POINTER(sz)]
    L.wt_open_times.argtypes = [vp, C.POINTER(OpenPhases)]
    L.wt_live.argtypes = [C.POINTER(LiveCounts)]
    L.wt_close.argtypes = [vp]
    L.wt_dlpack_file.argtypes = [C.c_char_p, C.c_int32, C.c_uint64, C.c_uint64, C.c_uint, C.POINTER(vp)]
    L.wt_dlpack_tensor.argtypes = [vp, sz, C.c_uint, C.POINTER(vp)]
    L.wt_dlpack_release.argtypes = [vp]
    L.wt_dlpack_live.argtypes = [C.POINTER(C.c_int64)]
    for s in SYMBOLS:
        if s not in ("wt_last_error", "wt_dlpack_release"):
            getattr(L, s).restype = C.c_int
    L.wt_dlpack_release.restype = None
    L.wt_last_error.restype = C.c_char_p
    _lib = L
    return L


def _check(rc: int):
    if rc != WT_OK:
        raise WtError(rc, lib().wt_last_error().decode(errors="replace"))


@dataclass(slots=True)
class TensorInfo:
    name: str
    dtype: int
    shape: Tuple[int, ...]
    nbytes: int
    file: int
    offset: int
    host_ptr: int


class OpenPhases(C.Structure):
    """wt_open_phases: wt_open's host time per hot-path step."""
    _fields_ = [("index_ms", C.c_double), ("index_cpu_ms", C.c_double), ("map_cpu_ms", C.c_double),
                ("prefault_ms", C.c_double), ("route_ms", C.c_double), ("files_mapped", C.c_uint64),
                ("files_registered", C.c_uint64)]


class TensorTable:
    """The index of an open checkpoint: TensorInfo per tensor, made on first access; the
    columns as plain lists (`names`, `dtypes`, `shapes`, `nbytes`, `files`, `offsets`,
    `host_ptrs`), each built on first use, for code that walks thousands of entries; and
    `meta`, the same columns as one numpy record array (META_DTYPE)."""

    def __init__(self, meta: np.ndarray, names: List[str]):
        self.meta = meta
        self.names = names
        self._items: List[object] = [None] * len(names)

    def _col(self, f):
        v = self.__dict__.get("_c_" + f)
        if v is None:
            v = self.__dict__["_c_" + f] = self.meta[f].tolist()
        return v

    dtypes = property(lambda self: self._col("dtype"))
    nbytes = property(lambda self: self._col("nbytes"))
    files = property(lambda self: self._col("file"))
    offsets = property(lambda self: self._col("offset"))
    host_ptrs = property(lambda self: self._col("host_ptr"))

    @property
    def shapes(self):
        v = self.__dict__.get("_c_shapes")
        if v is None:
            v = self.__dict__["_c_shapes"] = [tuple(sh[:nd]) for sh, nd in
                                              zip(self.meta["shape"].tolist(), self.meta["ndim"].tolist())]
        return v

    def __len__(self) -> int:
        return len(self.names)

    def __getitem__(self, i):
        if isinstance(i, slice):
            return [self[k] for k in range(*i.indices(len(self)))]
        t = self._items[i]
        if t is None:
            t = self._items[i] = TensorInfo(self.names[i], self.dtypes[i], self.shapes[i], self.nbytes[i],
                                            self.files[i], self.offsets[i], self.host_ptrs[i])
        return t

    def __iter__(self):
        return (self[i] for i in range(len(self)))


class Handle:
    """An open checkpoint (wt_open ... wt_close)."""

    def __init__(self, paths: Sequence[str], flags: int = 0):
        L = lib()
        # every path in one NUL-separated buffer, pointers computed from the NUL positions
        blob = ("\0".join(map(os.fspath, paths)) + "\0").encode() if len(paths) else b"\0"
        cbuf = C.create_string_buffer(blob, len(blob))
        ends = np.flatnonzero(np.frombuffer(blob, np.uint8) == 0)
        starts = np.concatenate(([0], ends[:-1] + 1)).astype(np.uint64) + np.uint64(C.addressof(cbuf))
        arr = np.ascontiguousarray(starts[:len(paths)] if len(paths) else np.zeros(1, np.uint64))
        h = C.c_void_p()
        _check(L.wt_open(C.cast(arr.ctypes.data, C.POINTER(C.c_char_p)), len(paths), flags, C.byref(h)))
        del cbuf, arr
        self._h = h
        self.flags = flags
        n = C.c_size_t()
        _check(L.wt_num_tensors(h, C.byref(n)))
        # two calls for the whole index (metadata table, then every name), not one per tensor
        meta = np.zeros(n.value, META_DTYPE)
        if n.value:
            _check(L.wt_tensor_table(h, 0, n.value, meta.ctypes.data))
        need = C.c_size_t()
        _check(L.wt_tensor_names(h, None, 0, C.byref(need)))
        buf = C.create_string_buffer(max(1, need.value))
        _check(L.wt_tensor_names(h, buf, need.value, C.byref(need)))
        names = buf.raw[:need.value].decode().split("\0")[:-1] if need.value else []
        self.tensors = TensorTable(meta, names)
        nf = C.c_size_t()
        _check(L.wt_num_files(h, C.byref(nf)))
        self.n_files = nf.value

    @property
    def ptr(self):
        if self._h is None:
            raise WtError(WT_EINVAL, "handle is closed")
        return self._h

    def find(self, name: str) -> int:
        i = C.c_size_t()
        _check(lib().wt_find(self.ptr, name.encode(), C.byref(i)))
        return i.value

    def route(self, f: int) -> int:
        r = C.c_uint()
        _check(lib().wt_file_route(self.ptr, f, C.byref(r)))
        return r.value

    def registration(self, f: int) -> int:
        """wt_file_registration: cudaHostRegister flags of file f (0 when not registered)."""
        r = C.c_uint()
        _check(lib().wt_file_registration(self.ptr, f, C.byref(r)))
        return r.value

    def adopt(self, idx: Sequence[int], dst: Sequence[int], mode: int = WT_ADOPT_GATHER,
              stream: int = 0, as_array: bool = False):
        """wt_adopt: returns the ready event (cudaEvent_t as int) of each tensor, as a list, or
        with as_array as a uint64 numpy array.  idx and dst may be numpy arrays."""
        ia = np.ascontiguousarray(idx, dtype=np.uint64).reshape(-1)
        da = np.ascontiguousarray(dst, dtype=np.uint64).reshape(-1)
        n = ia.size
        if da.size != n:
            raise ValueError("adopt: %d indices, %d destinations" % (n, da.size))
        if n == 0:
            ia = da = np.zeros(1, np.uint64)
        ra = np.zeros(max(1, n), np.uint64)
        _check(lib().wt_adopt(self.ptr, ia.ctypes.data, da.ctypes.data, n, mode, C.c_void_p(stream), ra.ctypes.data))
        return ra[:n] if as_array else ra[:n].tolist()

    def groups(self):
        """wt_tensor_groups: (group, block, n_groups): per tensor its logical tensor (uint32, in
        order of first appearance) and its row-block number (int32, -1 for a plain tensor)."""
        n = len(self.tensors)
        g, b = np.zeros(max(1, n), np.uint32), np.zeros(max(1, n), np.int32)
        ng = C.c_size_t()
        _check(lib().wt_tensor_groups(self.ptr, g.ctypes.data, b.ctypes.data, C.byref(ng)))
        return g[:n], b[:n], ng.value

    def pass_(self, descs, stream: int = 0):
        """wt_pass over a list of GemvDesc or a contiguous numpy array of DESC_DTYPE records."""
        if isinstance(descs, np.ndarray):
            if descs.dtype != DESC_DTYPE or not descs.flags.c_contiguous:
                raise ValueError("descriptor array must be a contiguous DESC_DTYPE array")
            n = descs.size
            arr = C.cast(descs.ctypes.data if n else 0, C.POINTER(GemvDesc))
        else:
            n = len(descs)
            arr = (GemvDesc * max(1, n))(*descs)
        _check(lib().wt_pass(self.ptr, arr, n, C.c_void_p(stream)))

    def checksum(self, ptrs: Sequence[int], nbytes: Sequence[int], out_dev: int, stream: int = 0,
                 plain: bool = False):
        n = len(ptrs)
        pa = (C.c_void_p * max(1, n))(*ptrs)
        na = (C.c_uint64 * max(1, n))(*nbytes)
        fn = lib().wt_checksum_plain if plain else lib().wt_checksum
        _check(fn(self.ptr, pa, na, n, C.c_void_p(out_dev), C.c_void_p(stream)))

    def device_status(self) -> int:
        s = C.c_int()
        _check(lib().wt_device_status(self.ptr, C.byref(s)))
        return s.value

    def residency(self) -> Tuple[int, int]:
        """wt_residency: (bytes resident in the page cache, total mapped bytes)."""
        r, t = C.c_uint64(), C.c_uint64()
        _check(lib().wt_residency(self.ptr, C.byref(r), C.byref(t)))
        return r.value, t.value

    def kernel_launches(self) -> int:
        v = C.c_uint64()
        _check(lib().wt_kernel_launches(self.ptr, C.byref(v)))
        return v.value

    def trace(self, origin_event: int) -> List[dict]:
        """wt_trace (WT_OPEN_TIMELINE handles): the ingest-batch and GEMV-group records, in
        enqueue order, with times in ms from `origin_event` (a cudaEvent_t with timing, e.g.
        ``torch.cuda.Event(enable_timing=True).cuda_event``).  Consumes the records."""
        n = C.c_size_t()
        cap = 1 << 16
        buf = (TraceRec * cap)()
        _check(lib().wt_trace(self.ptr, C.c_void_p(origin_event), buf, cap, C.byref(n)))
        kinds = {WT_TRACE_INGEST: "ingest", WT_TRACE_GEMV: "gemv"}
        return [dict(kind=kinds.get(buf[i].kind, "?"), index=buf[i].index, bytes=buf[i].bytes,
                     event=buf[i].event or 0, begin_ms=buf[i].begin_ms, end_ms=buf[i].end_ms)
                for i in range(min(n.value, cap))]

    def open_times(self) -> dict:
        """wt_open_times: host ms wt_open spent per step (index, map, prefault, route) and the
        counts of mapped and registered files."""
        o = OpenPhases()
        _check(lib().wt_open_times(self.ptr, C.byref(o)))
        return {f: getattr(o, f) for f, _ in OpenPhases._fields_}

    def pass_stamps(self):
        """wt_pass_stamps (WT_OPEN_STAMPS handles): the per-CTA stamps of the latest one-column
        GEMV launch, a uint64 array [grid, len(STAMP_FIELDS)] (nanoseconds but the "sm" column);
        empty before the first stamped launch.  Waits for the device."""
        import numpy as np
        n = C.c_size_t()
        _check(lib().wt_pass_stamps(self.ptr, None, 0, C.byref(n)))
        out = np.zeros((n.value, len(STAMP_FIELDS)), np.uint64)
        if n.value:
            _check(lib().wt_pass_stamps(self.ptr, C.c_void_p(out.ctypes.data), n.value, C.byref(n)))
        return out

    def close(self):
        if self._h is not None:
            h, self._h = self._h, None
            _check(lib().wt_close(h))

    def __enter__(self):
        return self

    def __exit__(self, *a):
        self.close()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def live() -> dict:
    """wt_live: handles, plans, events, device and pinned bytes the library has handed out
    now, and the bytes its block cache keeps for the next handle."""
    c = LiveCounts()
    _check(lib().wt_live(C.byref(c)))
    return {f: getattr(c, f) for f, _ in LiveCounts._fields_}


def checksum_noalloc(ptrs: Sequence[int], nbytes: Sequence[int], out_dev: int, stream: int = 0):
    """wt_checksum_noalloc: leaf-tree digests without any device allocation (no handle)."""
    n = len(ptrs)
    pa = (C.c_void_p * max(1, n))(*ptrs)
    na = (C.c_uint64 * max(1, n))(*nbytes)
    _check(lib().wt_checksum_noalloc(pa, na, n, C.c_void_p(out_dev), C.c_void_p(stream)))


def gemv_desc(W: int, dtype: int, M: int, K: int, x: int, y: int, wait_event: int = 0,
              scale: int = 0, cols: int = 0) -> GemvDesc:
    """One wt_gemv_desc; int8 weights (WT_I8) take fp16 x and `scale` = fp16 [M] row scales.
    cols = T in 1..16: x is X[T, K], y is Y[T, M] (the multi-column tensor-core kernel)."""
    return GemvDesc(W, dtype, cols, M, K, x, y, wait_event or None, scale or None)


# ----------------------------------------------------------------------------- DLPack producer

class DLDevice(C.Structure):
    _fields_ = [("device_type", C.c_int32), ("device_id", C.c_int32)]


class DLDataType(C.Structure):
    _fields_ = [("code", C.c_uint8), ("bits", C.c_uint8), ("lanes", C.c_uint16)]


class DLTensor(C.Structure):
    _fields_ = [("data", C.c_void_p), ("device", DLDevice), ("ndim", C.c_int32), ("dtype", DLDataType),
                ("shape", C.POINTER(C.c_int64)), ("strides", C.POINTER(C.c_int64)), ("byte_offset", C.c_uint64)]


class DLPackVersion(C.Structure):
    _fields_ = [("major", C.c_uint32), ("minor", C.c_uint32)]


class DLManagedTensorVersioned(C.Structure):
    _fields_ = [("version", DLPackVersion), ("manager_ctx", C.c_void_p), ("deleter", C.c_void_p),
                ("flags", C.c_uint64), ("dl_tensor", DLTensor)]


DLPACK_FLAG_BITMASK_READ_ONLY = 1
_CAPSULE_NAME = b"dltensor_versioned"  # must outlive every capsule: module constant
_capsule_new = C.pythonapi.PyCapsule_New
_capsule_new.restype = C.py_object
_capsule_new.argtypes = [C.c_void_p, C.c_char_p, C.c_void_p]
_capsule_is_valid = C.pythonapi.PyCapsule_IsValid
_capsule_is_valid.restype = C.c_int
_capsule_is_valid.argtypes = [C.c_void_p, C.c_char_p]
_capsule_get = C.pythonapi.PyCapsule_GetPointer
_capsule_get.restype = C.c_void_p
_capsule_get.argtypes = [C.c_void_p, C.c_char_p]


@C.CFUNCTYPE(None, C.c_void_p)
def _capsule_destructor(cap):
    # A capsule nobody adopted still carries its original name: run the producer's deleter.
    # A consumer renames the capsule it adopts and owns the deleter from then on.
    try:
        if _capsule_is_valid(cap, _CAPSULE_NAME):
            lib().wt_dlpack_release(_capsule_get(cap, _CAPSULE_NAME))
    except Exception:  # noqa: BLE001 - a destructor must not raise
        pass


class FileTensor:
    """One producer result (Algorithm 1): a read-only, file-backed DLManagedTensorVersioned
    awaiting adoption.  ``torch.from_dlpack(ft)`` makes a framework tensor over the file's
    pages with no copy; its storage then owns the mapping.  An instance exports once; if
    it is never exported, dropping it (or ``release()``) runs the deleter."""

    def __init__(self, ptr: int):
        self._p = ptr

    @classmethod
    def from_file(cls, path: str, dtype: int, M: int, K: int, flags: int = WT_DLPACK_DEVICE) -> "FileTensor":
        out = C.c_void_p()
        _check(lib().wt_dlpack_file(path.encode(), dtype, M, K, flags, C.byref(out)))
        return cls(out.value)

    @classmethod
    def from_handle(cls, h: "Handle", i: int, flags: int = WT_DLPACK_DEVICE) -> "FileTensor":
        out = C.c_void_p()
        _check(lib().wt_dlpack_tensor(h.ptr, i, flags, C.byref(out)))
        return cls(out.value)

    def _managed(self) -> DLManagedTensorVersioned:
        if self._p is None:
            raise BufferError("this FileTensor was already exported or released")
        return DLManagedTensorVersioned.from_address(self._p)

    @property
    def data_ptr(self) -> int:
        return self._managed().dl_tensor.data or 0

    @property
    def shape(self) -> Tuple[int, ...]:
        t = self._managed().dl_tensor
        return tuple(t.shape[k] for k in range(t.ndim))

    @property
    def strides(self) -> Tuple[int, ...]:
        t = self._managed().dl_tensor
        return tuple(t.strides[k] for k in range(t.ndim))

    @property
    def flags(self) -> int:
        return self._managed().flags

    @property
    def version(self) -> Tuple[int, int]:
        v = self._managed().version
        return (v.major, v.minor)

    def __dlpack_device__(self) -> Tuple[int, int]:
        d = self._managed().dl_tensor.device
        return (d.device_type, d.device_id)

    def __dlpack__(self, *, stream=None, max_version=None, dl_device=None, copy=None):
        """A "dltensor_versioned" capsule (DLPack 1.0, read-only flag set).  The pages hold no
        pending GPU work, so `stream` needs no synchronisation."""
        if max_version is None or tuple(max_version)[0] < 1:
            raise BufferError("the file-backed producer exports versioned (DLPack >= 1.0) capsules only")
        if copy:
            raise BufferError("the file-backed producer never copies")
        if dl_device is not None and tuple(dl_device) != self.__dlpack_device__():
            raise BufferError("the file-backed tensor lives on %s, not %s" % (self.__dlpack_device__(), tuple(dl_device)))
        p = self._p
        if p is None:
            raise BufferError("this FileTensor was already exported or released")
        cap = _capsule_new(p, _CAPSULE_NAME, C.cast(_capsule_destructor, C.c_void_p))
        self._p = None
        return cap

    def release(self):
        if self._p is not None:
            lib().wt_dlpack_release(self._p)
            self._p = None

    def __del__(self):
        try:
            self.release()
        except Exception:  # noqa: BLE001 - interpreter shutdown
            pass


def dlpack_live() -> int:
    n = C.c_int64()
    _check(lib().wt_dlpack_live(C.byref(n)))
    return n.value


def open(paths: Sequence[str], flags: int = 0) -> Handle:  # noqa: A001 - mirrors wt_open
    return Handle(paths, flags)
