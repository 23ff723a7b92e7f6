"""File -> first use, on top of the C ABI (torch supplies device memory and streams only).

    h = wt.Handle(paths)                       # wt_open: parse, map, route
    mats = matrices(h)                         # logical tensors as columns, row blocks joined
    dev = DeviceCheckpoint.allocate(h, mats)   # one caller-owned buffer per matrix/vector
    events = dev.adopt(h, mode, stream)        # wt_adopt: per-tensor ready events
    xs, ys = dev.inputs(), dev.outputs()       # x per inner size K, fp32 y per matrix
    h.pass_(dev.descs(xs, ys, events), stream) # wt_pass: each GEMV waits on its bytes only

The timed first use allocates while it ingests, with the step's inputs and outputs in the
first slab:

    x_host = host_inputs(mats)                                  # every x, pinned, once
    dev, events, _ = DeviceCheckpoint.stream_in(h, mats, mode, ingest, io=True)
    dev.io_x().copy_(x_host, non_blocking=True)                 # on the consumer stream
    h.pass_(dev.descs(dev.io_inputs(), dev.io_outputs(), events), consumer)

Row blocks: a tensor named "<name>#r<k>" is row block k of matrix <name> (the
many-small workload splits each matrix's rows across two files); its blocks are
adopted into one contiguous [M, K] device buffer, in k order, and the GEMV of
<name> waits on the event of its last-ingested block (the ingest stream is in
order, so that event implies the earlier blocks).  On a WT_OPEN_MAP_LARGE handle a
matrix whose blocks lie in both small (unmapped) and large (mapped) files crosses two
streams; it waits on an event recorded on the ingest stream after the wt_adopt call.
"""
from __future__ import annotations

from collections.abc import Mapping
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Sequence

import numpy as np

from . import synth, wt

_ESZ = {wt.WT_F32: 4, wt.WT_BF16: 2, wt.WT_F16: 2, wt.WT_I8: 1, wt.WT_U8: 1}
_ALIGN = 256


@dataclass(slots=True)
class MatrixRef:
    name: str
    dtype: int
    shape: tuple            # (M, K) for matrices, (n,) / other for non-GEMV tensors
    parts: List[int]        # tensor indices in row order
    gemv: bool              # 2-D with a GEMV dtype
    scale: Optional[int] = None  # tensor index of the fp16 row scales of int8 weights ("<name>.scale")


_GEMV_DT = (wt.WT_F32, wt.WT_BF16, wt.WT_F16)
_SMALL = 32  # checkpoints of at most this many tensors take the plain-loop branches
_GEMV_TAB = np.zeros(8, bool)  # dtype -> a GEMV dtype (int8 only with row scales)
_GEMV_TAB[list(_GEMV_DT)] = True


class Matrices:
    """The logical tensors of an open checkpoint (row blocks joined, wt_tensor_groups), in
    order of first appearance, as numpy columns: `dtype`, `M` and `K` (2-D and row-block
    tensors; 0 otherwise), `nbytes`, `gemv`, `scale` (tensor index of an int8 matrix's fp16 row
    scales, or -1) and the parts in CSR form (`part_ptr`, `part_idx`: tensor indices in
    block order).  A checkpoint of thousands of tensors is laid out, adopted and described to
    wt_pass from these columns; m[k] builds a MatrixRef on first access for code that wants
    one object per tensor."""

    def __init__(self, h: wt.Handle):
        T = h.tensors
        meta = T.meta
        group, block, ng = h.groups()
        self._names = T.names
        self._table = T
        self._refs: Dict[int, MatrixRef] = {}
        self._io = None
        n = len(group)
        if n <= _SMALL:
            self._init_small(T, group.tolist(), block.tolist(), ng)
            return
        if ng == n:  # no two tensors joined: logical tensor i is tensor i
            order = np.arange(n, dtype=np.int64)
            counts = np.ones(n, np.int64)
            ptr = np.arange(n + 1, dtype=np.int64)
        else:
            order = np.lexsort((block, group)).astype(np.int64)
            counts = np.bincount(group, minlength=ng).astype(np.int64)
            ptr = np.zeros(ng + 1, np.int64)
            np.cumsum(counts, out=ptr[1:])
        self.part_ptr, self.part_idx = ptr, order
        first = order[ptr[:-1]]
        self._first = first
        ndim = meta["ndim"].astype(np.int64)
        dt = meta["dtype"].astype(np.int64)
        shp = meta["shape"].astype(np.int64)
        self.stacked = block[first] >= 0
        two = (ndim[first] == 2) | self.stacked
        self.dtype = dt[first]
        self.K = np.where(two, shp[first, 1], 0)
        if bool(self.stacked.any()):
            # row blocks stack: 2-D, one dtype, one row length, distinct block numbers; each
            # part is compared with the first part of its logical tensor
            g_p = group[order]
            b_p = block[order]
            bad_p = (ndim[order] != 2) | (dt[order] != self.dtype[g_p]) | (shp[order, 1] != self.K[g_p])
            bad_p[1:] |= (b_p[1:] == b_p[:-1]) & (g_p[1:] == g_p[:-1])
            bad_p &= self.stacked[g_p]
            if bad_p.any():
                raise ValueError("row blocks of %s do not stack" % self.name(int(g_p[np.flatnonzero(bad_p)[0]])))
        if ng == n:
            self.M = np.where(two, shp[:, 0], 0)
            self.nbytes = meta["nbytes"].astype(np.int64)
        else:
            self.M = np.where(self.stacked, np.add.reduceat(shp[order, 0], ptr[:-1]), np.where(two, shp[first, 0], 0))
            self.nbytes = np.add.reduceat(meta["nbytes"].astype(np.int64)[order], ptr[:-1])
        self.gemv = two & _GEMV_TAB[np.minimum(self.dtype, 7)]
        self.scale = np.full(ng, -1, np.int64)
        self._find_scales(np.flatnonzero(two & (self.dtype == wt.WT_I8) & (counts == 1)).tolist())
        self.gemv_idx = np.flatnonzero(self.gemv)

    def _find_scales(self, q8: List[int]):
        """int8 matrices (2-D, one part) are GEMV matrices when their fp16 row scales, a 1-D
        tensor "<name>.scale" of M entries, are present."""
        if not q8:
            return
        T = self._table
        names = {nm: i for i, nm in enumerate(self._names)}
        for k in q8:
            si = names.get(self.name(k) + ".scale")
            if si is not None and T.dtypes[si] == wt.WT_F16 and T.shapes[si] == (int(self.M[k]),):
                self.scale[k] = si
                self.gemv[k] = True

    def _init_small(self, T, g: List[int], b: List[int], ng: int):
        """The same columns, for a checkpoint of a few tensors, with plain loops (a numpy call
        costs about as much as a loop over a few dozen entries)."""
        parts: List[List[tuple]] = [[] for _ in range(ng)]
        for i, (gi, bi) in enumerate(zip(g, b)):
            parts[gi].append((bi, i))
        dts, shs, nbs = T.dtypes, T.shapes, T.nbytes
        order, ptr, dtype, K, M, nbytes, two, stacked = [], [0], [], [], [], [], [], []
        for k, p in enumerate(parts):
            p.sort()
            idx = [i for _, i in p]
            f = idx[0]
            st = b[f] >= 0
            if st:
                blocks = [bi for bi, _ in p]
                if any(len(shs[i]) != 2 or dts[i] != dts[f] or shs[i][1] != shs[f][1] for i in idx) or \
                        len(set(blocks)) != len(blocks):
                    raise ValueError("row blocks of %s do not stack" % T.names[f].rpartition("#r")[0])
            t2 = st or len(shs[f]) == 2
            order += idx
            ptr.append(len(order))
            dtype.append(dts[f])
            K.append(shs[f][1] if t2 else 0)
            M.append(sum(shs[i][0] for i in idx) if st else (shs[f][0] if t2 else 0))
            nbytes.append(sum(nbs[i] for i in idx))
            two.append(t2)
            stacked.append(st)
        self.part_idx = np.asarray(order, np.int64)
        self.part_ptr = np.asarray(ptr, np.int64)
        self._first = self.part_idx[self.part_ptr[:-1]]
        self.stacked = np.asarray(stacked, bool)
        self.dtype = np.asarray(dtype, np.int64)
        self.K, self.M, self.nbytes = (np.asarray(v, np.int64) for v in (K, M, nbytes))
        self.gemv = np.asarray([t and d in _GEMV_DT for t, d in zip(two, dtype)], bool)
        self.scale = np.full(ng, -1, np.int64)
        self._find_scales([k for k in range(ng) if two[k] and dtype[k] == wt.WT_I8 and ptr[k + 1] - ptr[k] == 1])
        self.gemv_idx = np.flatnonzero(self.gemv)

    def __len__(self) -> int:
        return len(self.part_ptr) - 1

    def name(self, k: int) -> str:
        nm = self._names[int(self._first[k])]
        return nm.rpartition("#r")[0] if self.stacked[k] else nm

    def parts(self, k: int) -> List[int]:
        return self.part_idx[self.part_ptr[k]:self.part_ptr[k + 1]].tolist()

    def __getitem__(self, k):
        if isinstance(k, slice):
            return [self[i] for i in range(*k.indices(len(self)))]
        if k < 0:
            k += len(self)
        r = self._refs.get(k)
        if r is None:
            if self.stacked[k] or self.K[k]:
                shape = (int(self.M[k]), int(self.K[k]))
            else:
                shape = self._table.shapes[int(self._first[k])]
            sc = int(self.scale[k])
            r = self._refs[k] = MatrixRef(self.name(k), int(self.dtype[k]), shape, self.parts(k),
                                          bool(self.gemv[k]), sc if sc >= 0 else None)
        return r

    def __iter__(self):
        return (self[k] for k in range(len(self)))


def matrices(h: wt.Handle) -> Matrices:
    """Group the handle's tensors into logical tensors (row blocks joined), in first-seen order."""
    return Matrices(h)


def _matrices_list(h: wt.Handle) -> List[MatrixRef]:
    """The same grouping one tensor at a time, in plain Python: the reference the columnar
    grouping is tested against."""
    out: List[MatrixRef] = []
    by_name: Dict[str, MatrixRef] = {}
    blocks: Dict[str, Dict[int, int]] = {}
    gemv_dt = (wt.WT_F32, wt.WT_BF16, wt.WT_F16)
    T = h.tensors
    tnames, tdt, tshape = T.names, T.dtypes, T.shapes
    for i, nm in enumerate(tnames):
        base, sep, k = nm.rpartition("#r")
        if not sep or not k.isdigit() or not k.isascii() or len(k) > 9:
            sh = tshape[i]
            ref = MatrixRef(nm, tdt[i], sh, [i], len(sh) == 2 and tdt[i] in gemv_dt)
            out.append(ref)
            by_name[nm] = ref
            continue
        bl = blocks.get(base)
        if bl is None:
            bl = blocks[base] = {}
            if base not in by_name:
                ref = MatrixRef(base, tdt[i], (), [], False)
                out.append(ref)
                by_name[base] = ref
        bl[int(k)] = i
    for base, parts in blocks.items():
        ref = by_name[base]
        idx = [parts[k] for k in sorted(parts)]
        sh0, dt0 = tshape[idx[0]], tdt[idx[0]]
        K = sh0[1] if len(sh0) == 2 else None
        rows = 0
        for i in idx:
            sh = tshape[i]
            if K is None or len(sh) != 2 or sh[1] != K or tdt[i] != dt0:
                raise ValueError("row blocks of %s do not stack" % base)
            rows += sh[0]
        ref.parts = idx
        ref.shape = (rows, K)
        ref.gemv = dt0 in gemv_dt
    # int8 matrices are GEMV matrices when their fp16 row scales "<name>.scale" are present
    names = None
    for ref in out:
        if ref.dtype == wt.WT_I8 and len(ref.shape) == 2 and len(ref.parts) == 1:
            if names is None:
                names = {nm: i for i, nm in enumerate(tnames)}
            si = names.get(ref.name + ".scale")
            if si is not None and tdt[si] == wt.WT_F16 and tshape[si] == (ref.shape[0],):
                ref.scale, ref.gemv = si, True
    return out


class SlabViews:
    """Per logical tensor, a uint8 view of the slab that holds it, made on first access: a
    checkpoint of thousands of tensors needs their addresses (DeviceCheckpoint.ptrs) at once,
    but a torch view of each only when a caller reads one."""

    def __init__(self, spans):
        self._spans = spans  # (slab tensor, byte offset, bytes) per logical tensor
        self._views = {}

    def __len__(self):
        return len(self._spans)

    def __getitem__(self, k):
        v = self._views.get(k)
        if v is None:
            t, o, n = self._spans[k]
            v = self._views[k] = t[o:o + n]
        return v

    def __iter__(self):
        return (self[k] for k in range(len(self._spans)))


class FlatOutputs:
    """Every GEMV matrix's fp32 y in one device buffer (one D2H copy reads them all); y of
    matrix k starts `offset[k]` floats into it.  descs() takes the addresses from here without
    building a tensor per matrix."""

    def __init__(self, buf, ks, rows):
        self.buf = buf
        self.keys = ks if isinstance(ks, np.ndarray) and ks.dtype == np.int64 else np.asarray(ks, np.int64)
        self.rows = np.asarray(rows, np.int64)
        self.offs = np.zeros(self.keys.size, np.int64)
        if self.keys.size > 1:
            np.cumsum(self.rows[:-1], out=self.offs[1:])

    @property
    def offset(self) -> Dict[int, int]:
        return dict(zip(self.keys.tolist(), self.offs.tolist()))

    def _pos(self, ks):
        if ks is self.keys:
            return np.arange(ks.size)
        ks = np.asarray(ks, np.int64)
        j = np.searchsorted(self.keys, ks)
        if ks.size and (np.any(j >= self.keys.size) or np.any(self.keys[np.minimum(j, self.keys.size - 1)] != ks)):
            raise KeyError("no y for some of the matrices")
        return j

    def __getitem__(self, k):
        j = int(self._pos([k])[0])
        o = int(self.offs[j])
        return self.buf[o:o + int(self.rows[j])]

    def ptrs(self, ks) -> np.ndarray:
        return np.uint64(self.buf.data_ptr()) + (4 * self.offs[self._pos(ks)]).astype(np.uint64)


def io_layout(mats):
    """Byte layout of a step's inputs and outputs in one device region: the x of every distinct
    (K, dtype) of the GEMV matrices, each 256-byte aligned (int8 weights take fp16 x), then one
    fp32 y per GEMV matrix in gemv order.  Returns ({(K, dtype): (offset, nbytes)}, y offset,
    rows per GEMV matrix, total bytes)."""
    if isinstance(mats, Matrices):
        if mats._io is None and len(mats) <= _SMALL:
            xs, pos, rows = {}, 0, []
            for k in mats.gemv_idx.tolist():
                K, dt, M = int(mats.K[k]), int(mats.dtype[k]), int(mats.M[k])
                if (K, dt) not in xs:
                    n = K * (2 if dt == wt.WT_I8 else _ESZ[dt])
                    xs[(K, dt)] = (pos, n)
                    pos += -(-n // _ALIGN) * _ALIGN
                rows.append(M)
            mats._io = (xs, pos, rows, pos + 4 * sum(rows))
        if mats._io is None:
            g = np.flatnonzero(mats.gemv)
            key = mats.K[g] * 8 + mats.dtype[g]
            _, first = np.unique(key, return_index=True)
            xs, pos = {}, 0
            for j in np.sort(first).tolist():
                K, dt = int(mats.K[g[j]]), int(mats.dtype[g[j]])
                n = K * (2 if dt == wt.WT_I8 else _ESZ[dt])
                xs[(K, dt)] = (pos, n)
                pos += -(-n // _ALIGN) * _ALIGN
            rows = mats.M[g].tolist()
            mats._io = (xs, pos, rows, pos + 4 * int(mats.M[g].sum()))
        return mats._io
    xs, pos, rows = {}, 0, []
    for m in mats:
        if not m.gemv:
            continue
        key = (m.shape[1], m.dtype)
        if key not in xs:
            n = m.shape[1] * (2 if m.dtype == wt.WT_I8 else _ESZ[m.dtype])
            xs[key] = (pos, n)
            pos += -(-n // _ALIGN) * _ALIGN
        rows.append(m.shape[0])
    return xs, pos, rows, pos + 4 * sum(rows)


def host_inputs(mats):
    """A step's inputs on the host: every x of io_layout (N(0,1) from the seeded generator,
    cast to the weight dtype) packed in one pinned buffer with the device region's layout, so
    that one host-to-device copy moves them all."""
    import torch
    xs, y_off, _, _ = io_layout(mats)
    buf = torch.zeros(max(1, y_off), dtype=torch.uint8, pin_memory=True)
    for (K, dt), (o, n) in xs.items():
        buf[o:o + n] = torch.from_numpy(synth.make_x(K, dt))
    return buf


class ReadyEvents(Mapping):
    """The ready events of adopted tensors: `event[i]` (a cudaEvent_t as uint64, 0 = none) and
    `pos[i]`, tensor i's place in the order the tensors were handed to wt_adopt (-1 = not
    adopted).  A mapping tensor -> event, in that order, for code that walks it."""

    def __init__(self, n: int):
        self.event = np.zeros(n, np.uint64)
        self.pos = np.full(n, -1, np.int64)
        self.order = np.zeros(0, np.int64)

    def add(self, idx: np.ndarray, ev: np.ndarray):
        idx = np.asarray(idx, np.int64)
        self.event[idx] = ev
        self.pos[idx] = len(self.order) + np.arange(idx.size)
        self.order = np.concatenate((self.order, idx))

    def __getitem__(self, i):
        if self.pos[i] < 0:
            raise KeyError(i)
        return int(self.event[i])

    def __iter__(self):
        return iter(self.order.tolist())

    def __len__(self):
        return int(self.order.size)

    def last_of(self, tensors_ptr: np.ndarray, tensors: np.ndarray) -> np.ndarray:
        """Per group of `tensors` (CSR: group g is tensors[ptr[g]:ptr[g+1]], none empty) the
        event of its last-adopted tensor; KeyError if one was not adopted."""
        p = self.pos[tensors]
        if p.size and p.min() < 0:
            raise KeyError("a tensor of the pass was not adopted")
        mx = np.maximum.reduceat(p, tensors_ptr[:-1]) if p.size else p
        return self.event[self.order[mx]]


class TensorAddrs(Mapping):
    """Device address of each tensor adopted into a DeviceCheckpoint: a mapping tensor index ->
    address over one uint64 array (0 = none)."""

    def __init__(self, n: int):
        self.arr = np.zeros(n, np.uint64)

    def __getitem__(self, i):
        v = int(self.arr[i])
        if not v:
            raise KeyError(i)
        return v

    def __iter__(self):
        return iter(np.flatnonzero(self.arr).tolist())

    def __len__(self):
        return int(np.count_nonzero(self.arr))


def _inner_offsets(mats: Matrices, tnb: np.ndarray):
    """Per part (CSR order) its logical tensor and its byte offset inside it (the row blocks of
    a matrix follow one another in block order)."""
    if len(mats.part_idx) <= _SMALL:
        grp, inner = [], []
        pi, pp, t = mats.part_idx.tolist(), mats.part_ptr.tolist(), tnb.tolist()
        for k in range(len(pp) - 1):
            off = 0
            for j in range(pp[k], pp[k + 1]):
                grp.append(k)
                inner.append(off)
                off += t[pi[j]]
        return np.asarray(grp, np.int64), np.asarray(inner, np.int64)
    nb = tnb[mats.part_idx]
    cs = np.cumsum(nb) - nb
    counts = np.diff(mats.part_ptr)
    grp = np.repeat(np.arange(len(mats)), counts)
    return grp, cs - cs[mats.part_ptr[:-1]][grp] if nb.size else cs


def _aligned(n):
    return -(-n // _ALIGN) * _ALIGN


@dataclass
class DeviceCheckpoint:
    mats: Matrices
    bufs: object                         # per logical tensor a torch uint8 view (SlabViews or a list)
    dst: TensorAddrs = None              # tensor index -> device address
    canary: int = 0
    _tables: Dict[tuple, object] = field(default_factory=dict)
    ptrs: object = None                  # device address of each logical tensor's buffer (uint64 array)
    _joined: List[object] = field(default_factory=list)  # events of matrices that crossed two streams
    io: object = None  # with io=True: uint8 view of the inputs/outputs region (io_layout)

    def _set_dst(self, h: wt.Handle, a: int = 0, b: Optional[int] = None):
        """Addresses of the tensors of logical tensors [a, b) from their buffers' addresses."""
        m = self.mats
        b = len(m) if b is None else b
        pa, pb = int(m.part_ptr[a]), int(m.part_ptr[b])
        grp, inner = self._inner
        pi = m.part_idx[pa:pb]
        if pb - pa <= _SMALL:
            p, g, o = self.ptrs.tolist(), grp[pa:pb].tolist(), inner[pa:pb].tolist()
            self.dst.arr[pi] = [p[gi] + oi for gi, oi in zip(g, o)]
        else:
            self.dst.arr[pi] = self.ptrs[grp[pa:pb]] + inner[pa:pb].astype(np.uint64)
        return pi

    def _join_mixed(self, h: wt.Handle, a: int, b: int, events: ReadyEvents, mode: int, stream: int):
        """A matrix of [a, b) whose tensors took both ways of one WT_OPEN_MAP_LARGE wt_adopt call
        (mapped files on the device route, small unmapped files through the pinned ring on the
        library's own stream) has no tensor event that implies the others: all its tensors get
        one event recorded on `stream` after the call, which follows every byte of it."""
        if mode == wt.WT_ADOPT_STAGED or b <= a or not h.flags & wt.WT_OPEN_MAP_LARGE:
            return
        m = self.mats
        small = h.tensors.meta["host_ptr"] == 0
        pa, pb = int(m.part_ptr[a]), int(m.part_ptr[b])
        sp = small[m.part_idx[pa:pb]].astype(np.int64)
        p0 = m.part_ptr[a:b] - pa
        lo, hi = np.minimum.reduceat(sp, p0), np.maximum.reduceat(sp, p0)
        sc = m.scale[a:b]
        has = sc >= 0
        ssm = small[np.where(has, sc, 0)].astype(np.int64)
        lo = np.where(has, np.minimum(lo, ssm), lo)
        hi = np.where(has, np.maximum(hi, ssm), hi)
        mixed = np.flatnonzero(lo != hi) + a
        if not mixed.size:
            return
        import torch
        ev = torch.cuda.Event()
        ev.record(torch.cuda.ExternalStream(stream) if stream else torch.cuda.default_stream())
        self._joined.append(ev)
        for k in mixed.tolist():
            ts = m.parts(k) + ([int(m.scale[k])] if m.scale[k] >= 0 else [])
            events.event[ts] = ev.cuda_event

    @staticmethod
    def _new(h: wt.Handle, mats: Matrices, bufs, canary: int = 0) -> "DeviceCheckpoint":
        dc = DeviceCheckpoint(mats, bufs, TensorAddrs(len(h.tensors)), canary=canary,
                              ptrs=np.zeros(len(mats), np.uint64))
        dc._inner = _inner_offsets(mats, h.tensors.meta["nbytes"].astype(np.int64))
        return dc

    @staticmethod
    def allocate(h: wt.Handle, mats: Matrices, device="cuda", canary: int = 0,
                 slab: bool = True, io: bool = False) -> "DeviceCheckpoint":
        """One device buffer per logical tensor (optionally `canary` spare bytes after each).

        slab=True carves every buffer out of one allocation (256-byte aligned offsets); io=True
        (with slab) also puts the step's inputs and outputs (io_layout) at its start."""
        import torch
        sizes = mats.nbytes
        io_bytes = _aligned(io_layout(mats)[3]) if io and slab else 0
        if slab:
            al = _aligned(sizes + canary)
            offs = io_bytes + np.cumsum(al) - al
            pos = int(io_bytes + al.sum())
            big = torch.empty(max(pos, 1), dtype=torch.uint8, device=device)
            bufs = SlabViews([(big, o, n + canary) for o, n in zip(offs.tolist(), sizes.tolist())])
            dc = DeviceCheckpoint._new(h, mats, bufs, canary)
            dc.ptrs[:] = np.uint64(big.data_ptr()) + offs.astype(np.uint64)
            if io_bytes:
                dc.io = big[:io_bytes]
        else:
            bufs = [torch.empty(n + canary, dtype=torch.uint8, device=device) for n in sizes.tolist()]
            dc = DeviceCheckpoint._new(h, mats, bufs, canary)
            dc.ptrs[:] = [b.data_ptr() for b in bufs]
        dc._set_dst(h)
        return dc

    @staticmethod
    def stream_in(h: wt.Handle, mats: Matrices, mode: int = wt.WT_ADOPT_GATHER, stream: int = 0,
                  first_bytes: int = 256 << 20, growth: float = 2.0, device="cuda", io: bool = False):
        """Allocation (step 4) interleaved with ingest (step 5): the logical tensors are cut, at
        tensor boundaries and in order, into segments that start at about `first_bytes` and grow
        by `growth` each time; each segment gets its own device slab right before its wt_adopt
        call.  The link starts after the first small allocation, every later allocation (under
        0.2 ms per GB) runs while the previous, half as large segment crosses the link (about
        4.8 ms per GB), and the few, mostly large calls keep wt_adopt's batches large.  A
        checkpoint under 2 GB is one slab and one call.  io=True puts the step's inputs and
        outputs (io_layout) at the start of the first slab, so that they cost no allocation of
        their own.  Returns (DeviceCheckpoint, ReadyEvents, host seconds spent allocating)."""
        import time
        import torch
        sizes = mats.nbytes
        n = len(mats)
        bounds = segment_bounds(sizes, first_bytes, growth)
        spans = [None] * n
        dc = DeviceCheckpoint._new(h, mats, SlabViews(spans))
        events = ReadyEvents(len(h.tensors))
        alloc_s = 0.0
        io_bytes = _aligned(io_layout(mats)[3]) if io else 0
        for a, b in zip(bounds, bounds[1:]):
            t0 = time.perf_counter()
            al = _aligned(sizes[a:b])
            start = io_bytes if a == 0 else 0
            offs = start + np.cumsum(al) - al
            big = torch.empty(max(int(start + al.sum()), 1), dtype=torch.uint8, device=device)
            alloc_s += time.perf_counter() - t0
            if a == 0 and io_bytes:
                dc.io = big[:io_bytes]
            dc.ptrs[a:b] = np.uint64(big.data_ptr()) + offs.astype(np.uint64)
            for k, o, nb in zip(range(a, b), offs.tolist(), sizes[a:b].tolist()):
                spans[k] = (big, o, nb)
            idx = np.sort(dc._set_dst(h, a, b))
            if idx.size:
                events.add(idx, h.adopt(idx, dc.dst.arr[idx], mode, stream, as_array=True))
                dc._join_mixed(h, a, b, events, mode, stream)
        return dc, events, alloc_s

    def adopt(self, h: wt.Handle, mode: int = wt.WT_ADOPT_GATHER, stream: int = 0,
              order: Optional[Sequence[int]] = None) -> ReadyEvents:
        """wt_adopt every tensor (index order unless `order`); returns the ReadyEvents."""
        idx = np.asarray(order, np.int64) if order is not None else np.flatnonzero(self.dst.arr)
        events = ReadyEvents(len(h.tensors))
        if idx.size:
            events.add(idx, h.adopt(idx, self.dst.arr[idx], mode, stream, as_array=True))
        m = self.mats
        got = np.zeros(len(h.tensors), bool)
        got[idx] = True
        if len(m):
            whole = np.minimum.reduceat(got[m.part_idx].astype(np.int8), m.part_ptr[:-1]).astype(bool)
            # every logical tensor adopted whole is a run [a, b) of whole ones
            ks = np.flatnonzero(whole)
            if ks.size:
                breaks = np.flatnonzero(np.diff(ks) != 1)
                for lo, hi in zip(np.concatenate(([0], breaks + 1)), np.concatenate((breaks + 1, [ks.size]))):
                    self._join_mixed(h, int(ks[lo]), int(ks[hi - 1]) + 1, events, mode, stream)
        return events

    def io_inputs(self) -> Dict[tuple, int]:
        """Device address of each x in the io region, by (K, dtype), for descs()."""
        base = self.io.data_ptr()
        return {key: base + o for key, (o, _) in io_layout(self.mats)[0].items()}

    def io_x(self):
        """The x part of the io region (uint8), the destination of host_inputs' copy."""
        return self.io[:io_layout(self.mats)[1]]

    def io_outputs(self) -> FlatOutputs:
        """Every GEMV matrix's fp32 y in the io region, in gemv_mats() order."""
        import torch
        _, y_off, rows, total = io_layout(self.mats)
        buf = self.io[y_off:y_off + 4 * max(1, sum(rows))].view(torch.float32) if rows else \
            torch.empty(1, dtype=torch.float32, device=self.io.device)
        return FlatOutputs(buf, self.mats.gemv_idx, rows)

    def gemv_mats(self) -> List[int]:
        return self.mats.gemv_idx.tolist()

    def inputs(self, device="cuda") -> Dict[tuple, object]:
        """x per (K, dtype): N(0,1) from the seeded generator, cast to the weight dtype."""
        import torch
        return {key: torch.from_numpy(synth.make_x(*key)).to(device) for key in io_layout(self.mats)[0]}

    def outputs_flat(self, device="cuda") -> FlatOutputs:
        """One fp32 buffer holding every GEMV matrix's y, in gemv_mats() order."""
        import torch
        rows = io_layout(self.mats)[2]
        return FlatOutputs(torch.empty(max(1, sum(rows)), dtype=torch.float32, device=device), self.mats.gemv_idx, rows)

    def outputs(self, device="cuda") -> Dict[int, object]:
        import torch
        return {k: torch.empty(int(self.mats.M[k]), dtype=torch.float32, device=device)
                for k in self.gemv_mats()}

    def descs(self, xs, ys, events=None, only: Optional[Sequence[int]] = None) -> np.ndarray:
        """wt_pass descriptors (a DESC_DTYPE array) for the GEMV matrices, or for `only`.

        With `events` (ReadyEvents, or a mapping tensor -> event), matrix k waits on the event
        of its last-adopted row block (or of its row scales, if those came later)."""
        m = self.mats
        ks = m.gemv_idx if only is None else np.asarray(list(only), np.int64)
        if ks.size <= _SMALL:
            return self._descs_small(ks.tolist(), xs, ys, events)
        key = None if only is None else ks.tobytes()
        t = self._tables.get(key)
        if t is None:  # everything that depends only on this checkpoint's buffers and `ks`
            base = np.zeros(ks.size, wt.DESC_DTYPE)
            base["W"] = self.ptrs[ks]
            base["dtype"] = m.dtype[ks]
            base["M"] = m.M[ks]
            base["K"] = m.K[ks]
            sc = m.scale[ks]
            has = sc >= 0
            base["scale"] = np.where(has, self.dst.arr[np.maximum(sc, 0)], 0)
            xk = m.K[ks] * 8 + m.dtype[ks]
            if ks.size <= 64:  # few matrices: a dict beats np.unique's fixed cost
                first: Dict[int, int] = {}
                inv = np.asarray([first.setdefault(v, len(first)) for v in xk.tolist()], np.int64)
                uk = list(first)
            else:
                uk, inv = np.unique(xk, return_inverse=True)
                uk = uk.tolist()
            # per matrix, its tensors (parts, then the row scales) in CSR form
            cnt = m.part_ptr[ks + 1] - m.part_ptr[ks]
            if not has.any() and bool((cnt == 1).all()):  # one tensor per matrix
                tptr = np.arange(ks.size + 1, dtype=np.int64)
                ts = m.part_idx[m.part_ptr[ks]]
            else:
                tptr = np.zeros(ks.size + 1, np.int64)
                np.cumsum(cnt + has, out=tptr[1:])
                ts = np.empty(int(tptr[-1]), np.int64)
                seg = np.repeat(np.arange(ks.size), cnt)
                within = np.arange(seg.size) - np.repeat(np.cumsum(cnt) - cnt, cnt)
                ts[tptr[:-1][seg] + within] = m.part_idx[np.repeat(m.part_ptr[ks], cnt) + within]
                ts[tptr[1:][has] - 1] = sc[has]
            t = self._tables[key] = (base, [(u >> 3, u & 7) for u in uk], inv, tptr, ts)
        base, ukeys, inv, tptr, ts = t
        out = base.copy()
        if ks.size:
            xv = [xs[u] for u in ukeys]
            out["x"] = np.asarray([v if isinstance(v, int) else v.data_ptr() for v in xv], np.uint64)[inv]
        out["y"] = ys.ptrs(ks) if isinstance(ys, FlatOutputs) else [ys[k].data_ptr() for k in ks.tolist()]
        if events:
            if not isinstance(events, ReadyEvents):  # any mapping tensor -> event, in adoption order
                re = ReadyEvents(len(self.dst.arr))
                re.add(np.fromiter(events.keys(), np.int64), np.fromiter(events.values(), np.uint64))
                events = re
            out["wait_event"] = events.last_of(tptr, ts)
        return out

    def _descs_small(self, ks: List[int], xs, ys, events) -> np.ndarray:
        """descs() for a few matrices: the records built in a loop and converted once."""
        m = self.mats
        ptrs, dst = self.ptrs.tolist(), self.dst.arr
        if isinstance(ys, FlatOutputs):
            yp = ys.ptrs(ks).tolist()
        else:
            yp = [ys[k].data_ptr() for k in ks]
        if events and not isinstance(events, ReadyEvents):
            re = ReadyEvents(len(dst))
            re.add(np.fromiter(events.keys(), np.int64), np.fromiter(events.values(), np.uint64))
            events = re
        pos = events.pos.tolist() if events else None
        evs = events.event.tolist() if events else None
        recs = []
        for j, k in enumerate(ks):
            dt, M, K, sc = int(m.dtype[k]), int(m.M[k]), int(m.K[k]), int(m.scale[k])
            v = xs[(K, dt)]
            wait = 0
            if events:
                ts = m.part_idx[m.part_ptr[k]:m.part_ptr[k + 1]].tolist() + ([sc] if sc >= 0 else [])
                if min(pos[i] for i in ts) < 0:
                    raise KeyError("a tensor of the pass was not adopted")
                wait = evs[max(ts, key=pos.__getitem__)]
            recs.append((ptrs[k], dt, 0, M, K, v if isinstance(v, int) else v.data_ptr(), yp[j], wait,
                         int(dst[sc]) if sc >= 0 else 0))
        return np.array(recs, wt.DESC_DTYPE)

    def x_dtype(self, k) -> int:
        return wt.WT_F16 if self.mats.dtype[k] == wt.WT_I8 else int(self.mats.dtype[k])

    @property
    def weight_bytes(self) -> int:
        g = np.flatnonzero(self.mats.gemv)
        es = np.array([_ESZ.get(int(d), 0) for d in range(8)], np.int64)
        return int((self.mats.M[g] * self.mats.K[g] * es[self.mats.dtype[g]]).sum())

    @property
    def data_bytes(self) -> int:
        return int(self.mats.nbytes.sum())


def segment_bounds(sizes: np.ndarray, first_bytes: int = 256 << 20, growth: float = 2.0) -> List[int]:
    """stream_in's segments: logical tensors [bounds[j], bounds[j+1]).  A checkpoint under 2 GB
    is one segment; otherwise the first ends where the bytes so far reach `first_bytes`, and
    each later one ends where its own bytes reach `growth` times the previous target."""
    n = len(sizes)
    total = int(sizes.sum()) if n else 0
    seg = total if total < (2 << 30) else min(first_bytes, total)
    cs = np.cumsum(sizes)
    cuts, limit, lo = [], seg, 0
    while True:
        k = lo + int(np.searchsorted(cs[lo:], limit, side="left"))
        if k + 1 >= n:
            break
        lo = k + 1
        cuts.append(k + 1)
        seg = int(seg * growth)
        limit = int(cs[k]) + seg
    return [0] + cuts + [n]
