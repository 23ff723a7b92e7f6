"""The execution contract (Table "contract") and its ablation (Sec. 4), on CUDA.

  C1  adopt:  the GEMV reads the mapped file pages (the map endpoint).
      off:    per-use copy; every dispatch ingests its matrix into an HBM staging buffer
              (wt_adopt) and the GEMV waits on that copy's event.
  C2  retain: x and y stay in device memory across dispatches.
      off:    every dispatch takes x from a host array and hands y back to a host array
              (the activation round trip of a foreign dispatcher).
  C3  order on the GPU: dispatches are ordered in the framework stream.
      off:    the host drains the device before every dispatch.

A pass is one GEMV dispatch per matrix.  `excess` runs a pass behind an in-flight framework
workload (bf16 matmuls already queued on the framework stream) and reports the time added
over that workload alone, the quantity of Table "cube"(b) and of the ordering figure.
"""
from __future__ import annotations

import itertools
import statistics
import time

import numpy as np

from . import synth, wt

CELLS = [c for c in itertools.product((1, 0), repeat=3)]  # (C1, C2, C3)
ORDERINGS = ("stream", "event", "host_event", "drain")


def cell_name(c) -> str:
    return "%s, %s, %s" % ("map" if c[0] else "copy", "device" if c[1] else "round trip",
                           "stream" if c[2] else "drain")


class Contract:
    """Per-matrix dispatches over one checkpoint under any setting of C1, C2, C3."""

    def __init__(self, paths):
        import torch
        self.torch = torch
        self.h = wt.Handle(paths, wt.WT_OPEN_PREFAULT)
        self.idx = [i for i, t in enumerate(self.h.tensors) if len(t.shape) == 2]
        self.bytes = sum(self.h.tensors[i].nbytes for i in self.idx)
        self.staging = [torch.empty(self.h.tensors[i].nbytes, dtype=torch.uint8, device="cuda") for i in self.idx]
        self.x_host, self.x_dev, self.y_dev, self.y_host = [], [], [], []
        for i in self.idx:
            t = self.h.tensors[i]
            xb = torch.from_numpy(synth.make_x(t.shape[1], t.dtype))
            self.x_host.append(xb)                       # host array (pageable)
            self.x_dev.append(xb.cuda())
            self.y_dev.append(torch.empty(t.shape[0], dtype=torch.float32, device="cuda"))
            self.y_host.append(np.zeros(t.shape[0], np.float32))
        self.own = torch.cuda.Stream()
        torch.cuda.synchronize()

    def close(self):
        self.h.close()

    def _desc(self, n, W, ev=0):
        t = self.h.tensors[self.idx[n]]
        return wt.gemv_desc(W, t.dtype, t.shape[0], t.shape[1], self.x_dev[n].data_ptr(), self.y_dev[n].data_ptr(), ev)

    def dispatch(self, n, c1, c2, stream):
        """One GEMV of matrix n on `stream` under C1/C2 (C3 is the caller's ordering)."""
        torch = self.torch
        with torch.cuda.stream(stream):
            if not c2:
                self.x_dev[n].copy_(self.x_host[n])      # x arrives from a host array
            if c1:
                self.h.pass_([self._desc(n, self.h.tensors[self.idx[n]].host_ptr)], stream.cuda_stream)
            else:
                ev = self.h.adopt([self.idx[n]], [self.staging[n].data_ptr()], wt.WT_ADOPT_GATHER,
                                  stream.cuda_stream)[0]
                self.h.pass_([self._desc(n, self.staging[n].data_ptr(), ev)], stream.cuda_stream)
            if not c2:
                self.y_host[n] = self.y_dev[n].cpu().numpy()  # y back to a host array (waits for it)

    def run_pass(self, c1, c2, c3, stream=None):
        torch = self.torch
        stream = stream or torch.cuda.current_stream()
        for n in range(len(self.idx)):
            if not c3:
                torch.cuda.synchronize()                 # host-visible drain before the dispatch
            self.dispatch(n, c1, c2, stream)

    def run_ordered(self, mechanism, framework):
        """A C1 + C2 pass on our own stream, ordered after the framework stream by `mechanism`."""
        torch = self.torch
        for n in range(len(self.idx)):
            if mechanism == "stream":
                self.dispatch(n, 1, 1, framework)
                continue
            ev = torch.cuda.Event()
            ev.record(framework)
            if mechanism == "event":
                self.own.wait_event(ev)                  # cudaStreamWaitEvent: ordering stays on the GPU
            elif mechanism == "host_event":
                ev.synchronize()                         # cudaEventSynchronize: the host sees the signal
            elif mechanism == "drain":
                torch.cuda.synchronize()                 # every in-flight operation retires
            self.dispatch(n, 1, 1, self.own)

    def outputs(self, c2):
        return [self.y_host[n] if not c2 else self.y_dev[n].cpu().numpy() for n in range(len(self.idx))]


def framework_load(torch, n: int, size: int = 4096):
    """Queue n bf16 matmuls on the current stream: the in-flight framework workload."""
    a = torch.randn(size, size, device="cuda", dtype=torch.bfloat16)
    b = torch.randn(size, size, device="cuda", dtype=torch.bfloat16)
    def enqueue():
        c = None
        for _ in range(n):
            c = a @ b
        return c
    return enqueue


def _timed(torch, fn, reps):
    ts = []
    for _ in range(reps):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        fn()
        torch.cuda.synchronize()
        ts.append(time.perf_counter() - t0)
    return statistics.median(ts)


def measure(paths, reps: int = 5, load_ms: float = 20.0) -> dict:
    """Idle cube (GB/s per cell), loaded excess per condition removed, ordering mechanisms."""
    import torch
    c = Contract(paths)
    try:
        fw = torch.cuda.current_stream()
        out = {"working_set_bytes": c.bytes, "matrices": len(c.idx), "idle_gbs": {}, "excess_ms": {},
               "ordering_excess_ms": {}}
        for cell in CELLS:                                  # warm-up of every cell
            c.run_pass(*cell)
        torch.cuda.synchronize()
        for cell in CELLS:
            s = _timed(torch, lambda: c.run_pass(*cell), reps)
            out["idle_gbs"][cell_name(cell)] = round(c.bytes / s / 1e9, 2)
        # calibrate the in-flight load to about load_ms
        one = _timed(torch, framework_load(torch, 1), 3)
        n = max(1, int(load_ms / 1e3 / max(one, 1e-6)))
        load = framework_load(torch, n)
        base = _timed(torch, load, reps)
        out["load_ms"] = round(base * 1e3, 3)
        removals = {"C1+C2+C3": (1, 1, 1), "remove C3": (1, 1, 0), "remove C2": (1, 0, 1),
                    "remove C1": (0, 1, 1), "remove all": (0, 0, 0)}
        for name, cell in removals.items():
            s = _timed(torch, lambda: (load(), c.run_pass(*cell)), reps)
            out["excess_ms"][name] = round((s - base) * 1e3, 3)
        for mech in ORDERINGS:
            s = _timed(torch, lambda: (load(), c.run_ordered(mech, fw)), reps)
            out["ordering_excess_ms"][mech] = round((s - base) * 1e3, 3)
        return out
    finally:
        c.close()
