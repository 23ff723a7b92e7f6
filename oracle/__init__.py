"""CPU oracle (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the bench's CPU-baseline leg
import this package.  It wraps ``oracle.c`` (its own file reader, index
decoder, FNV-1a digests and fp64 GEMV) through ctypes and shares no code with
the CUDA library.  See ``oracle.c`` for the definitions and readings.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess
from typing import List, Optional, Sequence, Tuple

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "oracle.c")
LIB = os.path.join(HERE, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile liboracle.so next to its source (plain gcc, no fast-math, no FMA contraction)."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < os.path.getmtime(SRC):
        tmp = LIB + ".tmp.%d" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fno-fast-math",
                               "-ffp-contract=off", "-D_GNU_SOURCE", "-o", tmp, SRC, "-lm"])
        os.replace(tmp, LIB)
    return LIB


def lib():
    global _lib
    if _lib is None:
        build()
        L = C.CDLL(LIB)
        L.or_last_error.restype = C.c_char_p
        L.or_load.argtypes = [C.c_char_p, C.POINTER(C.c_void_p)]
        L.or_load.restype = C.c_int
        L.or_free.argtypes = [C.c_void_p]
        L.or_count.argtypes = [C.c_void_p]
        L.or_count.restype = C.c_uint32
        L.or_size.argtypes = [C.c_void_p]
        L.or_size.restype = C.c_uint64
        L.or_bytes.argtypes = [C.c_void_p]
        L.or_bytes.restype = C.c_void_p
        L.or_entry_info.argtypes = [C.c_void_p, C.c_uint32, C.POINTER(C.c_char_p),
                                    C.POINTER(C.c_int), C.POINTER(C.c_int),
                                    C.POINTER(C.c_uint64), C.POINTER(C.c_uint64),
                                    C.POINTER(C.c_uint64)]
        L.or_fnv1a64.argtypes = [C.c_void_p, C.c_uint64]
        L.or_fnv1a64.restype = C.c_uint64
        L.or_fnv_tree.argtypes = [C.c_void_p, C.c_uint64]
        L.or_fnv_tree.restype = C.c_uint64
        L.or_gemv.argtypes = [C.c_void_p, C.c_int, C.c_uint64, C.c_uint64, C.c_void_p,
                              C.c_void_p, C.c_void_p]
        L.or_gemv_rows.argtypes = [C.c_void_p, C.c_int, C.c_uint64, C.c_uint64, C.c_void_p,
                                   C.c_void_p, C.c_uint64, C.c_void_p, C.c_void_p]
        L.or_gemv_q8.argtypes = [C.c_void_p, C.c_void_p, C.c_uint64, C.c_uint64, C.c_void_p, C.c_void_p,
                                 C.c_uint64, C.c_void_p, C.c_void_p]
        _lib = L
    return _lib


class OracleError(RuntimeError):
    pass


class OracleFile:
    """A parsed checkpoint file held in host memory (O1)."""

    def __init__(self, path: str):
        L = lib()
        h = C.c_void_p()
        rc = L.or_load(path.encode(), C.byref(h))
        if rc != 0:
            raise OracleError(L.or_last_error().decode(errors="replace"))
        self._h = h
        self.path = path
        self.size = int(L.or_size(h))
        base = L.or_bytes(h)
        self.bytes = np.ctypeslib.as_array(C.cast(base, C.POINTER(C.c_uint8)), shape=(max(self.size, 1),))[:self.size]
        self.entries: List[dict] = []
        for i in range(L.or_count(h)):
            nm = C.c_char_p()
            dt, nd = C.c_int(), C.c_int()
            shp = (C.c_uint64 * 4)()
            off, nb = C.c_uint64(), C.c_uint64()
            L.or_entry_info(h, i, C.byref(nm), C.byref(dt), C.byref(nd), shp, C.byref(off), C.byref(nb))
            self.entries.append(dict(name=nm.value.decode(), dtype=dt.value,
                                     shape=tuple(int(shp[d]) for d in range(nd.value)),
                                     offset=int(off.value), nbytes=int(nb.value)))

    def blob(self, i: int) -> np.ndarray:
        e = self.entries[i]
        return self.bytes[e["offset"]:e["offset"] + e["nbytes"]]

    def close(self):
        if self._h:
            lib().or_free(self._h)
            self._h = None
            self.bytes = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def load(path: str) -> OracleFile:
    return OracleFile(path)


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data if a.size else 0


def fnv1a64(data) -> int:
    """D_plain: literal FNV-1a-64 of the bytes (O2)."""
    a = np.ascontiguousarray(np.frombuffer(bytes(data), np.uint8) if isinstance(data, (bytes, bytearray)) else data).view(np.uint8)
    return int(lib().or_fnv1a64(_ptr(a), a.size))


def fnv_tree(data) -> int:
    """D_tree: FNV-1a-64 over LE64(n) and the LE64 digests of 4096-byte leaves (O2)."""
    a = np.ascontiguousarray(np.frombuffer(bytes(data), np.uint8) if isinstance(data, (bytes, bytearray)) else data).view(np.uint8)
    return int(lib().or_fnv_tree(_ptr(a), a.size))


def gemv(W: np.ndarray, dtype: int, M: int, K: int, x: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """(yhat, a): y = W x and sum |W_ij x_j| in fp64 (O3).  W, x are raw element bytes."""
    W = np.ascontiguousarray(W).view(np.uint8)
    x = np.ascontiguousarray(x).view(np.uint8)
    yhat = np.zeros(M, np.float64)
    a = np.zeros(M, np.float64)
    if M and lib().or_gemv(_ptr(W), dtype, M, K, _ptr(x), _ptr(yhat), _ptr(a)) != 0:
        raise OracleError("gemv: bad dtype")
    return yhat, a


def gemv_rows(W: np.ndarray, dtype: int, M: int, K: int, x: np.ndarray,
              rows: Sequence[int]) -> Tuple[np.ndarray, np.ndarray]:
    W = np.ascontiguousarray(W).view(np.uint8)
    x = np.ascontiguousarray(x).view(np.uint8)
    r = np.ascontiguousarray(rows, dtype=np.uint64)
    yhat = np.zeros(r.size, np.float64)
    a = np.zeros(r.size, np.float64)
    if r.size and lib().or_gemv_rows(_ptr(W), dtype, M, K, _ptr(x), _ptr(r), r.size,
                                     _ptr(yhat), _ptr(a)) != 0:
        raise OracleError("gemv_rows: bad dtype or row")
    return yhat, a


def gemv_q8(W: np.ndarray, s: np.ndarray, M: int, K: int, x: np.ndarray,
            rows: Optional[Sequence[int]] = None) -> Tuple[np.ndarray, np.ndarray]:
    """(yhat, a) for int8 W [M, K] with fp16 row scales s [M] and fp16 x [K] (O3, int8 form):
    yhat_i = s_i * sum_j W_ij x_j, a_i = |s_i| * sum_j |W_ij x_j|; all rows or the given rows."""
    W = np.ascontiguousarray(W).view(np.uint8)
    s = np.ascontiguousarray(s).view(np.uint8)
    x = np.ascontiguousarray(x).view(np.uint8)
    r = None if rows is None else np.ascontiguousarray(rows, dtype=np.uint64)
    n = M if r is None else r.size
    yhat = np.zeros(n, np.float64)
    a = np.zeros(n, np.float64)
    if n and lib().or_gemv_q8(_ptr(W), _ptr(s), M, K, _ptr(x), None if r is None else _ptr(r), n,
                              _ptr(yhat), _ptr(a)) != 0:
        raise OracleError("gemv_q8: bad row")
    return yhat, a


def gemv_cols(W: np.ndarray, dtype: int, M: int, K: int, X: np.ndarray, T: int,
              scale: Optional[np.ndarray] = None,
              rows: Optional[Sequence[int]] = None) -> Tuple[np.ndarray, np.ndarray]:
    """(Yhat, A), each [T, n], for the multi-column GEMV of the T-sweep (Sec. 4.3): X holds T
    activation vectors as rows of [T, K] (fp16 for int8 weights, else W's dtype) and column t
    of the result is the one-column GEMV of X[t]:  Yhat[t] = diag(scale) W X[t] (scale only
    for int8 weights, dtype 3), A[t] = the matching sum of |products|.  All rows or `rows`."""
    X = np.ascontiguousarray(X).view(np.uint8).reshape(-1)
    xes = 2 if dtype == 3 else {0: 4, 1: 2, 2: 2}[dtype]
    if X.size != T * K * xes:
        raise OracleError("gemv_cols: X holds %d bytes, want T*K*%d = %d" % (X.size, xes, T * K * xes))
    n = M if rows is None else len(rows)
    Y = np.zeros((T, n), np.float64)
    A = np.zeros((T, n), np.float64)
    for t in range(T):
        xt = X[t * K * xes:(t + 1) * K * xes]
        if dtype == 3:
            Y[t], A[t] = gemv_q8(W, scale, M, K, xt, rows=rows)
        elif rows is None:
            Y[t], A[t] = gemv(W, dtype, M, K, xt)
        else:
            Y[t], A[t] = gemv_rows(W, dtype, M, K, xt, rows)
    return Y, A


def gemv_error(y: np.ndarray, yhat: np.ndarray, a: np.ndarray) -> float:
    """max_i |y_i - yhat_i| / a_i; a row with a_i = 0 must give y_i == 0 exactly (else inf)."""
    y = np.asarray(y, np.float64)
    zero = a == 0
    if np.any(y[zero] != 0):
        return float("inf")
    nz = ~zero
    if not np.any(nz):
        return 0.0
    return float(np.max(np.abs(y[nz] - yhat[nz]) / a[nz]))


class CheckpointOracle:
    """All files of one checkpoint, parsed by the oracle; matrices assembled by name."""

    def __init__(self, paths: Sequence[str]):
        self.files = [load(p) for p in paths]

    def entry(self, f: int, i: int) -> dict:
        return self.files[f].entries[i]

    def digests(self) -> List[List[Tuple[int, int]]]:
        """Per file, per entry: (D_plain, D_tree)."""
        out = []
        for fo in self.files:
            out.append([(fnv1a64(fo.blob(i)), fnv_tree(fo.blob(i))) for i in range(len(fo.entries))])
        return out

    def find(self, name: str) -> Tuple[int, int]:
        for f, fo in enumerate(self.files):
            for i, e in enumerate(fo.entries):
                if e["name"] == name:
                    return f, i
        raise KeyError(name)

    def blob_of(self, f: int, name: str) -> np.ndarray:
        """Bytes of the entry `name` of file `f` (names are unique within a file only)."""
        fo = self.files[f]
        return fo.blob([e["name"] for e in fo.entries].index(name))

    def matrix_bytes(self, parts: Sequence[Tuple[int, str]]) -> np.ndarray:
        """Row blocks given as (file, name), in row order, concatenated (the many workload's halves)."""
        blobs = [self.blob_of(f, n) for f, n in parts]
        return blobs[0] if len(blobs) == 1 else np.concatenate(blobs)

    def close(self):
        for fo in self.files:
            fo.close()
