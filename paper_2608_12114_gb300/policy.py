"""Endpoint selection at deployment (Algorithm 2, Sec. 8.1), measured on GB300.

A weight byte reaches the GEMV by one of three endpoints:

  map       the GEMV reads the file pages in place over the host link (wt_pass with W
            inside the handle's mapping; contract C1, no second copy)
  resident  one copy into HBM, amortised over every pass; the GEMV streams HBM
  copy      per-use copy: each pass ingests the pages into an HBM staging buffer
            (wt_adopt) and the GEMV of each batch starts on its event (overlapped streaming)

Algorithm 2 maps the working set W and prefaults it; stops with "storage-bound" when the
mapped set is not resident; measures B_map over the full mapped set; builds a resident arm
holding all of W (dropped when the allocation fails or the mapping is evicted after one
pass of every arm); measures B_dev and B_copy with the same kernel and set; ranks the
endpoints by W/B and, when the leaders lie within the band theta, chooses map (one
evictable file-backed representation instead of a second owned copy).
"""
from __future__ import annotations

import statistics
import time
from dataclasses import dataclass, field
from typing import Callable, Dict, Optional

THETA = 0.05  # the paper's tie band (5 %)
ENDPOINTS = ("map", "resident", "copy")


def select(times_ms: Dict[str, Optional[float]], theta: float = THETA) -> str:
    """Algorithm 2's last two steps: rank the surviving endpoints by W/B (ms) and, if the
    mapped endpoint lies within `theta` of the leader, choose it.

    Returns "map" (map leads), "map (tie)" (map within the band of the leader),
    "resident" or "copy".  Dropped endpoints are absent or None.  The band is relative to
    the mapped endpoint's own time: (t_map - t_best) / t_map <= theta, i.e. the leader's
    rate exceeds map's by at most theta of itself."""
    live = {k: v for k, v in times_ms.items() if v is not None}
    if not live:
        raise ValueError("no endpoint survived")
    best = min(live, key=live.get)
    if best == "map":
        return "map"
    if "map" in live and (live["map"] - live[best]) / live["map"] <= theta:
        return "map (tie)"
    return best


@dataclass
class PolicyResult:
    working_set_bytes: int
    resident_before: int
    resident_after: Optional[int]
    rates_gbs: Dict[str, Optional[float]] = field(default_factory=dict)
    times_ms: Dict[str, Optional[float]] = field(default_factory=dict)
    dropped: Dict[str, str] = field(default_factory=dict)
    decision: str = ""
    theta: float = THETA

    def as_dict(self) -> dict:
        return dict(working_set_bytes=self.working_set_bytes, resident_before=self.resident_before,
                    resident_after=self.resident_after, rates_gbs=self.rates_gbs, times_ms=self.times_ms,
                    dropped=self.dropped, decision=self.decision, theta=self.theta)


def run(working_set_bytes: int, residency: Callable[[], tuple], measure: Dict[str, Callable[[], Optional[float]]],
        theta: float = THETA) -> PolicyResult:
    """Algorithm 2 over measured arms.

    residency()        -> (resident bytes, total bytes) of the mapped set (wt_residency)
    measure[endpoint]  -> seconds for one pass over W at that endpoint, or a string saying
                          why the arm cannot be built (e.g. the resident allocation failed)
    The map arm is measured first (over the full mapped set), then resident, then copy;
    residency is queried again after one pass of every arm."""
    res0, tot = residency()
    out = PolicyResult(working_set_bytes, res0, None, theta=theta)
    if res0 < tot:
        out.decision = "storage-bound"
        out.dropped = {e: "mapped set not resident" for e in ENDPOINTS}
        return out
    for e in ENDPOINTS:
        s = measure[e]()
        if s is None or isinstance(s, str):
            out.dropped[e] = s or "arm could not be built"
            out.rates_gbs[e], out.times_ms[e] = None, None
        else:
            out.rates_gbs[e] = working_set_bytes / s / 1e9
            out.times_ms[e] = s * 1e3
    res1, tot1 = residency()
    out.resident_after = res1
    if res1 < tot1 and out.times_ms.get("resident") is not None:
        out.dropped["resident"] = "mapping evicted after one pass of every arm"
        out.times_ms["resident"] = None
    out.decision = select(out.times_ms, theta)
    return out


def median_pass_seconds(run_pass: Callable[[], None], sync: Callable[[], None], reps: int = 5,
                        warmup: int = 1) -> float:
    """Median wall time of `reps` passes (each synchronised), after `warmup` passes."""
    for _ in range(warmup):
        run_pass()
        sync()
    ts = []
    for _ in range(reps):
        t0 = time.perf_counter()
        run_pass()
        sync()
        ts.append(time.perf_counter() - t0)
    return statistics.median(ts)


def measure_gb300(paths, reps: int = 5, theta: float = THETA) -> PolicyResult:
    """Algorithm 2 on this GPU for the checkpoint `paths` (torch supplies memory and streams)."""
    import torch

    from . import pipeline, wt

    h = wt.Handle(paths, wt.WT_OPEN_PREFAULT)  # map at deployed granularity; prefault
    try:
        mats = pipeline.matrices(h)
        gm = [k for k, m in enumerate(mats) if m.gemv]
        wbytes = sum(h.tensors[i].nbytes for k in gm for i in mats[k].parts)
        xs = {}
        for k in gm:
            m = mats[k]
            key = (m.shape[1], m.dtype)
            if key not in xs:
                from . import synth
                xs[key] = torch.from_numpy(synth.make_x(m.shape[1], m.dtype)).cuda()
        ys = {k: torch.empty(mats[k].shape[0], dtype=torch.float32, device="cuda") for k in gm}
        s = torch.cuda.Stream()
        sync = s.synchronize

        # map: W is the mapping itself (row blocks of one matrix must be adjacent in one file)
        def measure_map():
            descs = []
            for k in gm:
                m = mats[k]
                parts = [h.tensors[i] for i in m.parts]
                if any(p.file != parts[0].file for p in parts) or any(
                        b.offset != a.offset + a.nbytes for a, b in zip(parts, parts[1:])):
                    return "a matrix's row blocks are not one contiguous mapped range"
                descs.append(wt.gemv_desc(parts[0].host_ptr, m.dtype, m.shape[0], m.shape[1],
                                          xs[(m.shape[1], m.dtype)].data_ptr(), ys[k].data_ptr()))
            return median_pass_seconds(lambda: h.pass_(descs, s.cuda_stream), sync, reps)

        holder = {}

        def build_resident():
            try:
                dev = pipeline.DeviceCheckpoint.allocate(h, mats)
            except torch.OutOfMemoryError:
                return "allocation of the resident copy failed (capacity)"
            dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
            sync()
            holder["dev"] = dev
            return dev

        def measure_resident():
            dev = build_resident()
            if isinstance(dev, str):
                return dev
            d = dev.descs(xs, ys)
            return median_pass_seconds(lambda: h.pass_(d, s.cuda_stream), sync, reps)

        def measure_copy():
            dev = holder.get("dev") or build_resident()
            if isinstance(dev, str):
                return "no HBM staging buffer: " + dev

            def one():
                ev = dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
                h.pass_(dev.descs(xs, ys, ev), s.cuda_stream)
            return median_pass_seconds(one, sync, reps)

        return run(wbytes, h.residency, {"map": measure_map, "resident": measure_resident, "copy": measure_copy},
                   theta)
    finally:
        h.close()
