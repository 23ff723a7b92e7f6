"""File -> first use, on top of the C ABI (torch supplies device memory and streams only).

    h = wt.Handle(paths)                       # wt_open: parse, map, route
    mats = matrices(h)                         # 2-D tensors, row blocks joined
    dev = DeviceCheckpoint.allocate(h, mats)   # one caller-owned buffer per matrix/vector
    events = dev.adopt(h, mode, stream)        # wt_adopt: per-tensor ready events
    xs, ys = dev.inputs(), dev.outputs()       # x per inner size K, fp32 y per matrix
    h.pass_(dev.descs(xs, ys, events), stream) # wt_pass: each GEMV waits on its bytes only

Row blocks: a tensor named "<name>#r<k>" is row block k of matrix <name> (the
many-small workload splits each matrix's rows across two files); its blocks are
adopted into one contiguous [M, K] device buffer, in k order, and the GEMV of
<name> waits on the event of its last-ingested block (the ingest stream is in
order, so that event implies the earlier blocks).  On a WT_OPEN_MAP_LARGE handle a
matrix whose blocks lie in both small (unmapped) and large (mapped) files crosses two
streams; it waits on an event recorded on the ingest stream after the wt_adopt call.
"""
from __future__ import annotations

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


def matrices(h: wt.Handle) -> List[MatrixRef]:
    """Group the handle's tensors into logical tensors (row blocks joined), in first-seen order."""
    out: List[MatrixRef] = []
    by_name: Dict[str, MatrixRef] = {}
    blocks: Dict[str, Dict[int, int]] = {}
    gemv_dt = (wt.WT_F32, wt.WT_BF16, wt.WT_F16)
    T = h.tensors
    tnames, tdt, tshape = T.names, T.dtypes, T.shapes
    for i, nm in enumerate(tnames):
        base, sep, k = nm.rpartition("#r")
        if not sep or not k.isdigit() or not k.isascii():
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

    def __init__(self, buf, offset: Dict[int, int]):
        self.buf = buf
        self.offset = offset

    def __getitem__(self, k):
        return self.buf[self.offset[k]:self.offset[k] + self._rows[k]]

    def ptrs(self, ks) -> np.ndarray:
        base = self.buf.data_ptr()
        return base + 4 * np.fromiter((self.offset[k] for k in ks), np.uint64, len(ks))


@dataclass
class DeviceCheckpoint:
    mats: List[MatrixRef]
    bufs: object                         # per MatrixRef a torch uint8 view (SlabViews or a list)
    dst: Dict[int, int] = field(default_factory=dict)  # tensor index -> device address
    canary: int = 0
    _tables: Dict[tuple, object] = field(default_factory=dict)
    ptrs: List[int] = field(default_factory=list)  # device address of each MatrixRef's buffer
    _joined: List[object] = field(default_factory=list)  # events of matrices that crossed two streams

    def _join_mixed(self, h: wt.Handle, ks: Sequence[int], events: Dict[int, int], mode: int, stream: int):
        """A matrix of `ks` whose tensors took both ways of one WT_OPEN_MAP_LARGE wt_adopt call
        (mapped files on the device route, small unmapped files through the pinned ring on the
        library's own stream) has no tensor event that implies the others: all its tensors get
        one event recorded on `stream` after the call, which follows every byte of it."""
        if mode == wt.WT_ADOPT_STAGED:
            return
        hp = h.tensors.host_ptrs
        mixed = []
        for k in ks:
            ts = self.mats[k].parts + ([self.mats[k].scale] if self.mats[k].scale is not None else [])
            if len({hp[i] == 0 for i in ts}) > 1:
                mixed.append(ts)
        if not mixed:
            return
        import torch
        ev = torch.cuda.Event()
        ev.record(torch.cuda.ExternalStream(stream) if stream else torch.cuda.default_stream())
        self._joined.append(ev)
        for ts in mixed:
            for i in ts:
                events[i] = ev.cuda_event

    @staticmethod
    def allocate(h: wt.Handle, mats: Sequence[MatrixRef], device="cuda", canary: int = 0,
                 slab: bool = True) -> "DeviceCheckpoint":
        """One device buffer per logical tensor (optionally `canary` spare bytes after each).

        slab=True carves every buffer out of one allocation (256-byte aligned offsets)."""
        import torch
        tnb = h.tensors.nbytes
        sizes = [sum(tnb[i] for i in m.parts) for m in mats]
        if slab:
            offs, pos = [], 0
            for n in sizes:
                offs.append(pos)
                pos += -(-(n + canary) // _ALIGN) * _ALIGN
            big = torch.empty(max(pos, 1), dtype=torch.uint8, device=device)
            bufs = SlabViews([(big, o, n + canary) for o, n in zip(offs, sizes)])
            base = big.data_ptr()
            ptrs = [base + o for o in offs]
        else:
            bufs = [torch.empty(n + canary, dtype=torch.uint8, device=device) for n in sizes]
            ptrs = [b.data_ptr() for b in bufs]
        dc = DeviceCheckpoint(list(mats), bufs, canary=canary, ptrs=ptrs)
        for m, p in zip(mats, ptrs):
            off = 0
            for i in m.parts:
                dc.dst[i] = p + off
                off += tnb[i]
        return dc

    @staticmethod
    def stream_in(h: wt.Handle, mats: Sequence[MatrixRef], mode: int = wt.WT_ADOPT_GATHER, stream: int = 0,
                  first_bytes: int = 256 << 20, growth: float = 2.0, device="cuda"):
        """Allocation (step 4) interleaved with ingest (step 5): the logical tensors are cut, at
        tensor boundaries and in order, into segments that start at about `first_bytes` and grow
        by `growth` each time; each segment gets its own device slab right before its wt_adopt
        call.  The link starts after the first small allocation, every later allocation (under
        0.2 ms per GB) runs while the previous, half as large segment crosses the link (about
        4.8 ms per GB), and the few, mostly large calls keep wt_adopt's batches large.  A
        checkpoint under 2 GB is one slab and one call.  Returns (DeviceCheckpoint,
        tensor -> ready event, host seconds spent allocating)."""
        import time
        import torch
        tnb = h.tensors.nbytes
        sizes = [sum(tnb[i] for i in m.parts) for m in mats]
        total = sum(sizes)
        seg = total if total < (2 << 30) else min(first_bytes, total)
        cuts, acc, limit = [], 0, seg
        for k, n in enumerate(sizes):
            acc += n
            if acc >= limit and k + 1 < len(sizes):
                cuts.append(k + 1)
                seg = int(seg * growth)
                limit = acc + seg
        bounds = [0] + cuts + [len(mats)]
        spans = [None] * len(mats)
        dc = DeviceCheckpoint(list(mats), SlabViews(spans), ptrs=[0] * len(mats))
        events: Dict[int, int] = {}
        alloc_s = 0.0
        for a, b in zip(bounds, bounds[1:]):
            t0 = time.perf_counter()
            offs, pos = [], 0
            for k in range(a, b):
                offs.append(pos)
                pos += -(-sizes[k] // _ALIGN) * _ALIGN
            big = torch.empty(max(pos, 1), dtype=torch.uint8, device=device)
            alloc_s += time.perf_counter() - t0
            base = big.data_ptr()
            idx = []
            for k, o in zip(range(a, b), offs):
                spans[k] = (big, o, sizes[k])
                dc.ptrs[k] = p = base + o
                off = 0
                for i in mats[k].parts:
                    dc.dst[i] = p + off
                    off += tnb[i]
                    idx.append(i)
            idx.sort()
            if idx:
                events.update(zip(idx, h.adopt(idx, [dc.dst[i] for i in idx], mode, stream)))
                dc._join_mixed(h, range(a, b), events, mode, stream)
        return dc, events, alloc_s

    def adopt(self, h: wt.Handle, mode: int = wt.WT_ADOPT_GATHER, stream: int = 0,
              order: Optional[Sequence[int]] = None) -> Dict[int, int]:
        """wt_adopt every tensor (file/index order unless `order`); returns tensor -> event."""
        idx = list(order) if order is not None else sorted(self.dst)
        evs = dict(zip(idx, h.adopt(idx, [self.dst[i] for i in idx], mode, stream)))
        got = set(idx)
        self._join_mixed(h, [k for k, m in enumerate(self.mats) if got.issuperset(m.parts)], evs, mode, stream)
        return evs

    def gemv_mats(self) -> List[int]:
        return [k for k, m in enumerate(self.mats) if m.gemv]

    def inputs(self, device="cuda") -> Dict[tuple, object]:
        """x per (K, dtype): N(0,1) from the seeded generator, cast to the weight dtype."""
        import torch
        xs = {}
        for k in self.gemv_mats():
            m = self.mats[k]
            key = (m.shape[1], m.dtype)
            if key not in xs:
                xs[key] = torch.from_numpy(synth.make_x(m.shape[1], m.dtype)).to(device)
        return xs

    def outputs_flat(self, device="cuda") -> FlatOutputs:
        """One fp32 buffer holding every GEMV matrix's y, in gemv_mats() order."""
        import torch
        ks = self.gemv_mats()
        rows = [self.mats[k].shape[0] for k in ks]
        offs = np.concatenate(([0], np.cumsum(rows)[:-1])).astype(np.int64).tolist() if ks else []
        fo = FlatOutputs(torch.empty(max(1, sum(rows)), dtype=torch.float32, device=device), dict(zip(ks, offs)))
        fo._rows = dict(zip(ks, rows))
        return fo

    def outputs(self, device="cuda") -> Dict[int, object]:
        import torch
        return {k: torch.empty(self.mats[k].shape[0], dtype=torch.float32, device=device)
                for k in self.gemv_mats()}

    def descs(self, xs, ys, events: Optional[Dict[int, int]] = None,
              only: Optional[Sequence[int]] = None) -> np.ndarray:
        """wt_pass descriptors (a DESC_DTYPE array) for the GEMV matrices, or for `only`.

        With `events`, matrix k waits on the event of its last-ingested row block."""
        ks = list(only) if only is not None else self.gemv_mats()
        key = tuple(ks)
        base = self._tables.get(key)
        if base is None:  # the parts that depend only on this checkpoint's buffers
            base = np.zeros(len(ks), wt.DESC_DTYPE)
            mats = [self.mats[k] for k in ks]
            base["W"] = [self.ptrs[k] for k in ks]
            base["dtype"] = [m.dtype for m in mats]
            base["M"] = [m.shape[0] for m in mats]
            base["K"] = [m.shape[1] for m in mats]
            base["scale"] = [self.dst[m.scale] if m.scale is not None else 0 for m in mats]
            self._tables[key] = base
        out = base.copy()
        out["x"] = [xs[(self.mats[k].shape[1], self.mats[k].dtype)].data_ptr() for k in ks]
        out["y"] = ys.ptrs(ks) if isinstance(ys, FlatOutputs) else [ys[k].data_ptr() for k in ks]
        if events:
            pos = {i: n for n, i in enumerate(events)}
            out["wait_event"] = [events[max(self.mats[k].parts + ([self.mats[k].scale] if self.mats[k].scale is not None else []),
                                            key=pos.__getitem__)] for k in ks]
        return out

    def x_dtype(self, k) -> int:
        return wt.WT_F16 if self.mats[k].dtype == wt.WT_I8 else self.mats[k].dtype

    @property
    def weight_bytes(self) -> int:
        return sum(int(np.prod(self.mats[k].shape)) * _ESZ[self.mats[k].dtype] for k in self.gemv_mats())

    @property
    def data_bytes(self) -> int:
        return sum(int(np.prod(m.shape)) * _ESZ[m.dtype] for m in self.mats)
