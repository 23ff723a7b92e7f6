"""Benchmark of the file-backed weight path on GB300 (one JSON line on stdout).

Metric: file -> first-use ingest GB/s, and resident GEMV-pass GB/s against HBM peak.

  value   resident pass: every matrix of the checkpoint through the persistent
          TMA-fed GEMV (one launch per pass), weights already in HBM; weight
          bytes / time (the paper's convention: weight bytes counted once).
  e2e     file -> first use through the C ABI: wt_open (parse, map, route),
          wt_adopt (host-mapped pages -> HBM, per-batch events), the
          event-gated first GEMV pass, and the device -> host read of every y;
          ingested data bytes / wall time.  Page cache warm (the paper's
          precondition for adoption).

A step is one resident pass over the whole checkpoint.  Inputs (16 GB for the
default workload) are far larger than L2, so no flush is needed between passes.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload large|mid|many|sweep:I|tiny]
  python bench.py --impl reference ...   # the CPU oracle on a bounded sample (the reference arm)
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "file→first-use ingest GB/s; resident GEMV-pass GB/s vs HBM peak (%)"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0

WORKLOADS = {
    "large": "large decoder checkpoint, bf16, 4 shards (16.06 GB): 32 layers, d=4096, kv 1024, FFN 14336, vocab 128256",
    "mid": "mid decoder checkpoint, bf16, 3 shards (5.40 GB): 32 layers, d=2560, FFN 6912, vocab 32000",
    "many": "many-small: 1253 bf16 matrices split by rows across 2506 files (1.56 GB)",
    "tiny": "tiny: 8 fp32 256x256 matrices + 8 fp32[256] vectors in one file (2.1 MB)",
    "protocol": "matched protocol by bytes: 12 files of one bf16 12288x3584 matrix (88.1 MB each, 1.06 GB)",
    "protocol_q8": "matched protocol: 12 files of one int8 12288x7168 matrix (88.1 MB) + fp16 row scales; fp16 x",
}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=400, help="timed resident passes")
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", default="wt", choices=["wt", "reference"])
    p.add_argument("--workload", default="large")
    p.add_argument("--layers", type=int, default=None, help="override decoder layer count (small profiling cases)")
    p.add_argument("--mode", default="gather", choices=["gather", "ce", "staged"])
    p.add_argument("--open", default="map", choices=["map", "nomap", "prefault", "register", "maplarge"],
                   help="nomap: wt_open maps nothing (WT_OPEN_NOMAP) and --mode staged preads into the pinned ring; "
                        "prefault: wt_open populates every mapping (WT_OPEN_PREFAULT); maplarge: only files of at "
                        "least WT_MAP_MIN_BYTES are mapped, the rest adopted through the pinned ring "
                        "(WT_OPEN_MAP_LARGE)")
    p.add_argument("--e2e-reps", type=int, default=5)
    p.add_argument("--skip-e2e", action="store_true", help="resident passes only (profiling runs)")
    p.add_argument("--arms", action="store_true", help="also time the ce/staged/stock-torch ingest arms")
    p.add_argument("--graph", action="store_true",
                   help="time the resident pass as replays of one captured CUDA graph")
    p.add_argument("--stamps", action="store_true",
                   help="after the timed region, per-CTA stamps of the resident pass (WT_OPEN_STAMPS): "
                        "prologue, plan-table reads, first copy, streaming, tail")
    p.add_argument("--graph-passes", type=int, default=1,
                   help="with --graph: resident passes captured in the graph (steps rounds up to a multiple)")
    p.add_argument("--cold-reps", type=int, default=0,
                   help="also time N file -> first-use runs with the files evicted from the page cache")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=15.0, help="CPU budget of the oracle sample")
    p.add_argument("--ref-seconds", type=float, default=150.0,
                   help="total CPU budget of the reference arm (--impl reference), split over its steps")
    p.add_argument("--data-dir", default=None)
    p.add_argument("--workers", type=int, default=0)
    p.add_argument("--cube", action="store_true",
                   help="the C1/C2/C3 contract ablation and ordering mechanisms on the protocol workload")
    p.add_argument("--tsweep", default=None, metavar="T,T,...",
                   help="multi-column T-sweep (e.g. 0,1,2,4,8,16; 0 = the one-column kernel) on the "
                        "int8 matched protocol by default (one JSON line)")
    p.add_argument("--checksum", action="store_true",
                   help="time wt_checksum (leaf-tree FNV-1a-64) over every resident tensor of the workload")
    p.add_argument("--consumer-priority", default="high", choices=["high", "normal"],
                   help="priority of the stream the event-gated first-use GEMVs run on")
    p.add_argument("--fresh", action="store_true",
                   help="with --timeline: allocate the device buffers inside each traced run (step 4), "
                        "as the e2e value does")
    p.add_argument("--timeline", action="store_true",
                   help="one traced file -> first-use run (WT_OPEN_TIMELINE): per ingest batch and GEMV group, "
                        "device begin/end times (one JSON line)")
    p.add_argument("--policy", action="store_true",
                   help="measure the map / resident / per-use-copy endpoints and apply Algorithm 2 (one JSON line)")
    return p.parse_args()


# ----------------------------------------------------------------------------- workload files

def workload_ck(args, outdir):
    from paper_2608_12114_gb300 import synth
    w = args.workload
    if w.startswith("sweep:"):
        return synth.sweep(outdir, points=[int(w.split(":")[1])])
    if w == "tiny":
        return synth.tiny(outdir)
    if w == "protocol":
        return synth.protocol(outdir)
    if w == "protocol_q8":
        return synth.protocol_q8(outdir)
    if w == "many":
        return synth.many(outdir)
    if w in ("mid", "large"):
        return synth.decoder(outdir, w, layers=args.layers)
    raise SystemExit("unknown workload " + w)


DT_NAME = {0: "f32", 1: "bf16", 2: "f16", 3: "int8"}
L2_BYTES = 129 * 10 ** 6  # GB300 L2
DATA_DESC = {
    "bf16": "synthetic (seeded N(0,0.02) bf16 weights, norms 1.0, x ~ N(0,1))",
    "int8": "synthetic (seeded uniform int8 weights in [-127, 127], fp16 row scales, fp16 x ~ N(0,1))",
}


def gemv_alg_bytes(dtype, M, K):
    """Bytes one GEMV must move at minimum: W once, x once, y once (+ the fp16 row scales
    of int8 weights, whose activations are fp16)."""
    es = {0: 4, 1: 2, 2: 2, 3: 1}[dtype]
    xes = 2 if dtype == 3 else es
    return M * K * es + K * xes + 4 * M + (2 * M if dtype == 3 else 0)


def workload_desc(args):
    w = args.workload
    if w.startswith("sweep:"):
        i = int(w.split(":")[1])
        return "size sweep point %d: one bf16 4096x%d matrix (%d MiB)" % (i, 128 << i, 1 << i)
    d = WORKLOADS[w]
    if args.layers is not None:
        d += " (reduced to %d layers)" % args.layers
    return d


def make_files(args, rank, world):
    """Rank 0 writes the workload (spawned workers, before any CUDA call); all ranks share it."""
    from paper_2608_12114_gb300 import synth
    base = args.data_dir or os.path.join(tempfile.gettempdir(), "wt_bench")
    outdir = os.path.join(base, args.workload.replace(":", "_") + ("_l%d" % args.layers if args.layers else ""))
    ck = workload_ck(args, outdir)
    t0 = time.time()
    if rank == 0:
        workers = args.workers or min(16, os.cpu_count() or 1)
        synth.write_files(ck, workers=workers)
        os.sync()
    gen_s = time.time() - t0
    return ck, gen_s


# ----------------------------------------------------------------------------- measurement helpers

class Clocks:
    """nvidia-smi samples of SM clock and throttle reasons, taken while the timed region runs."""

    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, bus_id):
        self.bus_id = bus_id
        self.p = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        cmd = ["nvidia-smi", "--query-gpu=" + self.Q, "--format=csv,noheader,nounits", "-lms", "50"]
        if self.bus_id:
            cmd += ["-i", self.bus_id]
        try:
            self.p = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None
        time.sleep(0.5)
        self.t0 = time.time()
        return self

    def __exit__(self, *a):
        self.t1 = time.time()
        if self.p:
            time.sleep(0.15)
            self.p.terminate()
            self.p.wait()

    def summary(self):
        import datetime
        rows = []
        if self.path and os.path.exists(self.path):
            for line in open(self.path):
                f = [x.strip() for x in line.split(",")]
                if len(f) < 9:
                    continue
                try:
                    ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                except ValueError:
                    continue
                if self.t0 - 0.05 <= ts <= self.t1 + 0.05:
                    rows.append(f)
            os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        def num(v):
            try:
                return float(v)
            except ValueError:
                return None
        sm = [num(r[1]) for r in rows if num(r[1]) is not None]
        mx = [num(r[2]) for r in rows if num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9]) if v.strip().lower() == "active"})
        pw = [num(r[3]) for r in rows if num(r[3]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None}


def bus_id():
    try:
        import torch
        pr = torch.cuda.get_device_properties(torch.cuda.current_device())
        return "%08X:%02X:%02X.0" % (pr.pci_domain_id, pr.pci_bus_id, pr.pci_device_id)
    except Exception:
        return None


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        try:
            d = json.load(open(p))
            return float(d["hbm_gbs"]), "measured"
        except Exception:
            pass
    return FALLBACK_HBM_GBS, "fallback"


def pinned_h2d_gbs(torch, nbytes=1 << 30, reps=10):
    """Copy-engine H2D from a pinned (cudaMallocHost) buffer, best of `reps`: the ingest roofline."""
    return h2d_probe(torch, nbytes, reps, streams=(1,), sm_loads=False)["ce_1_stream"]


def h2d_probe(torch, nbytes=1 << 30, reps=10, streams=(1, 2, 4), sm_loads=True):
    """Host -> device ceilings over the host link, best of `reps` each, GB/s:
    ce_<n>_stream  the copy engines moving one pinned 1 GiB buffer cut into n equal parts, one
                   cudaMemcpyAsync per part on n concurrent streams (timed from an event before
                   the first to one after the last, all on the device);
    sm_loads       the map-endpoint GEMV kernel reading the same pinned buffer as a bf16 matrix
                   in place (16-byte loads from every SM, full occupancy): the link as SM loads
                   see it, with the kernel's own arithmetic on top."""
    from paper_2608_12114_gb300 import wt
    h = torch.empty(nbytes, dtype=torch.uint8, pin_memory=True)
    h.fill_(1)
    d = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    out = {}
    for n in streams:
        ss = [torch.cuda.Stream() for _ in range(n)]
        part = nbytes // n
        best = 1e30
        for _ in range(reps):
            torch.cuda.synchronize()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(ss[0])
            for k, st in enumerate(ss[1:], 1):
                st.wait_event(a)
            for k, st in enumerate(ss):
                with torch.cuda.stream(st):
                    d[k * part:(k + 1) * part].copy_(h[k * part:(k + 1) * part], non_blocking=True)
            for st in ss[1:]:
                ev = torch.cuda.Event()
                ev.record(st)
                ss[0].wait_event(ev)
            b.record(ss[0])
            b.synchronize()
            best = min(best, a.elapsed_time(b))
        out["ce_%d_stream" % n] = round(n * part / best / 1e6, 1)
    if sm_loads:
        K = 8192
        M = nbytes // (2 * K)
        y = torch.empty(M, dtype=torch.float32, device="cuda")
        x = torch.ones(K, dtype=torch.bfloat16, device="cuda")
        s = torch.cuda.Stream()
        with wt.Handle([]) as hh:
            desc = [wt.gemv_desc(h.data_ptr(), wt.WT_BF16, M, K, x.data_ptr(), y.data_ptr())]
            hh.pass_(desc, s.cuda_stream)
            s.synchronize()
            best = 1e30
            for _ in range(max(3, reps // 2)):
                a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                a.record(s)
                hh.pass_(desc, s.cuda_stream)
                b.record(s)
                b.synchronize()
                best = min(best, a.elapsed_time(b))
            if hh.device_status() != 0:
                raise SystemExit("device status %d in the H2D probe" % hh.device_status())
        out["sm_loads"] = round(M * K * 2 / best / 1e6, 1)
        del y, x
    del h, d
    return out


def int8_tc_kernel(ms, T):
    """The tensor-core kernel an int8 launch of matrices ms ([(M, K)]) with T columns runs:
    the row-owner kernel when its 128-row blocks number at least two per CTA slot (or when
    WT_COLS_KERNEL=q8rows), else the warp-MMA kernel (as the library decides)."""
    force = os.environ.get("WT_COLS_KERNEL")
    blocks = sum(-(-M // 128) for M, _ in ms)
    if force == "q8rows" or (force != "mma" and blocks >= 2 * 152):
        return "gemm_q8_rows_kernel<NT=%d> (mma.sync m16n8k16, row-owner warps)" % (2 if T > 8 else 1)
    return "gemm_cols_kernel<int8, NT=%d> (mma.sync m16n8k16)" % (2 if T > 8 else 1)


def onecol_kernel_name(wdt, ms):
    """The kernel a one-column resident pass runs: the TMA GEMV, or for int8 rows up to
    K = 8192 a tensor-core kernel at T = 1 (unless WT_I8_ONECOL=cuda)."""
    if wdt == "int8" and os.environ.get("WT_I8_ONECOL") != "cuda" and max(K for _, K in ms) <= 8192:
        return int8_tc_kernel(ms, 1)
    return "gemv_tma_kernel<%s>" % wdt


def kernel_source_digest():
    """First 16 hex digits of the SHA-256 over the GEMV kernel's sources (kernel file, shared
    device helpers, tile geometry header): a captured traffic figure is valid only for them."""
    h = hashlib.sha256()
    for f in ("wt_kernels.cu", "wt_device.cuh", "wt_kernels.h"):
        h.update(open(os.path.join(ROOT, "paper_2608_12114_gb300", "csrc", f), "rb").read())
    return h.hexdigest()[:16]


def kernel_traffic(name):
    """DRAM bytes per launch from the committed ncu summary, if it matches the current kernels."""
    p = os.path.join(ROOT, "profiles", name)
    if not os.path.exists(p):
        return None
    try:
        d = json.load(open(p))
    except Exception:
        return None
    digest = kernel_source_digest()
    if d.get("kernel_source_sha256_16") != digest:
        return None
    return d


# ----------------------------------------------------------------------------- replicas (N > 1)

def combine_ranks(dist, device, total_ms, e2e_s):
    """Max over ranks of the timed-region length and of the first-use time: the slowest
    replica sets the clock.  Without a process group the local values are returned."""
    if dist is None:
        return total_ms, e2e_s
    import torch
    t = torch.tensor([total_ms, e2e_s], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return tuple(t.tolist())


def aggregate_gbs(bytes_per_rank, world, seconds):
    """Whole-job rate: every replica moves the same bytes, the job takes the slowest time."""
    return bytes_per_rank * world / seconds / 1e9


# ----------------------------------------------------------------------------- the wt arm

def stamp_summary(wt, st):
    """Medians over the CTAs with rows of each stamp, in us from the CTA's own entry, plus the
    launch's span (first entry to last exit) and the spread of the CTAs' entries."""
    import numpy as np
    F = {f: i for i, f in enumerate(wt.STAMP_FIELDS)}
    t = st.astype(np.int64)
    busy = t[t[:, F["first_copy"]] > 0]
    rel = lambda f: round(float(np.median(busy[:, F[f]] - busy[:, F["entry"]])) / 1e3, 3)
    return {"ctas": int(t.shape[0]), "ctas_with_rows": int(busy.shape[0]),
            "median_us_from_entry": {f: rel(f) for f in wt.STAMP_FIELDS[1:-1]},
            "span_us": round(float(t[:, F["exit"]].max() - t[:, F["entry"]].min()) / 1e3, 3),
            "entry_spread_us": round(float(t[:, F["entry"]].max() - t[:, F["entry"]].min()) / 1e3, 3),
            "first_copy_to_last_full_us_median": round(float(np.median(busy[:, F["last_full"]] - busy[:, F["first_copy"]])) / 1e3, 3)}


def run_stamps(torch, wt, descs, s, args, gp):
    """The resident pass on a WT_OPEN_STAMPS handle (outside the timed region): the stamps of
    the last of `warmup` + 20 host-issued passes and, with --graph, of the last pass of the last
    replay of a graph of gp passes."""
    out = {"what": "per-CTA %globaltimer stamps of the stamping instantiation of the resident kernel, "
                   "medians over the CTAs with rows, us from each CTA's entry (prologue: mbarriers ready; "
                   "operands: past the wait for the previous grid; first_copy: first bulk copy issued, after "
                   "the plan-table reads; first_full / last_full: first / last stage landed; exit)"}
    with wt.Handle([], wt.WT_OPEN_STAMPS) as hs:
        for _ in range(args.warmup + 20):
            hs.pass_(descs, s.cuda_stream)
        s.synchronize()
        out["host_issued"] = stamp_summary(wt, hs.pass_stamps())
        if args.graph:
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=s):
                for _ in range(gp):
                    hs.pass_(descs, torch.cuda.current_stream().cuda_stream)
            with torch.cuda.stream(s):
                for _ in range(args.warmup + 5):
                    g.replay()
            s.synchronize()
            out["graph"] = stamp_summary(wt, hs.pass_stamps())
            out["graph"]["passes_per_graph"] = gp
            del g
        if hs.device_status() != 0:
            raise SystemExit("device status %d after stamped passes" % hs.device_status())
    return out


def open_flags(wt, name):
    return {"map": 0, "nomap": wt.WT_OPEN_NOMAP, "prefault": wt.WT_OPEN_PREFAULT,
            "register": wt.WT_ROUTE_REGISTER, "maplarge": wt.WT_OPEN_MAP_LARGE}[name]


def consumer_stream(torch, args):
    """The stream of the event-gated GEMVs.  At high priority the block scheduler places a
    GEMV group's CTAs before those of the gather batch that becomes ready at the same moment."""
    if args.consumer_priority == "high":
        return torch.cuda.Stream(priority=-1)
    return torch.cuda.Stream()


def make_slab(torch, pipeline, h, mats, dev=None, x_host=None):
    """Step 4, device allocation: one torch slab for the checkpoint (256-byte aligned views;
    or `dev`, already allocated with its io region) whose first bytes hold the step's inputs
    and outputs: the x of every inner size and one fp32 y per matrix (pipeline.io_layout).
    With `x_host` (pipeline.host_inputs) the x region is filled from it before returning."""
    if dev is None:
        dev = pipeline.DeviceCheckpoint.allocate(h, mats, io=True)
    ys = dev.io_outputs()
    sl = {"dev": dev, "xs": dev.io_inputs(), "ys": ys, "yflat": ys.buf, "xdev": dev.io_x()}
    if x_host is not None:
        sl["xdev"].copy_(x_host)
        torch.cuda.synchronize()
    return sl


def first_use(torch, wt, pipeline, ck, mode, ingest_s, consume_s, x_host, y_host, slab, phases=None, flags=0,
              trace=None):
    """One file -> first-use run; returns (seconds, handle stats).  `slab` None allocates the
    device buffers inside the timed run (step 4), after the previous run's memory went back to
    the driver; otherwise the given buffers are reused.  The step's inputs (every x, in the
    pinned `x_host`) cross to the device inside the run, and every y comes back to the pinned
    `y_host`.  With `phases` (a dict), also records
    host-side phase times in ms: open (wt_open: parse, map, route), alloc (device buffers, x,
    y), enqueue (wt_adopt + wt_pass return; includes page-table population), drain (until y is
    on the host), and the route of the first file.  With `trace` (a list; the handle is then
    opened with WT_OPEN_TIMELINE), the run's ingest/GEMV records are appended to it."""
    if slab is None:
        torch.cuda.empty_cache()
        torch.cuda.synchronize()
    origin = torch.cuda.Event(enable_timing=True) if trace is not None else None
    t0 = time.perf_counter()
    h = wt.Handle(ck.paths, flags | (wt.WT_OPEN_TIMELINE if trace is not None else 0))
    mats = pipeline.matrices(h)
    t1 = time.perf_counter()
    ot = h.open_times() if phases is not None else None
    if origin is not None:
        origin.record(ingest_s)
    if slab is None:
        # allocation interleaved with ingest: a small first slab, then the rest segment by
        # segment while earlier bytes cross the link; x and y once the link is busy
        dev, ev, alloc_s = pipeline.DeviceCheckpoint.stream_in(h, mats, mode, ingest_s.cuda_stream, io=True)
        tx = time.perf_counter()
        sl = make_slab(torch, pipeline, h, mats, dev)
        alloc_s += time.perf_counter() - tx
    else:
        sl, alloc_s = slab, 0.0
        dev = sl["dev"]
        ev = dev.adopt(h, mode, ingest_s.cuda_stream)
    ta = t1 + alloc_s
    with torch.cuda.stream(consume_s):
        sl["xdev"].copy_(x_host, non_blocking=True)
        h.pass_(dev.descs(sl["xs"], sl["ys"], ev), consume_s.cuda_stream)
        y_host.copy_(sl["yflat"], non_blocking=True)
    t2 = time.perf_counter()
    consume_s.synchronize()
    dt = time.perf_counter() - t0
    if phases is not None:
        phases.setdefault("open_ms", []).append((t1 - t0) * 1e3)
        phases.setdefault("alloc_ms", []).append(alloc_s * 1e3)
        phases.setdefault("enqueue_ms", []).append((t2 - t1 - alloc_s) * 1e3)
        phases.setdefault("drain_ms", []).append((t0 + dt - t2) * 1e3)
        phases["route"] = wt.ROUTE_NAMES.get(h.route(0), "?") if h.n_files else None
        for k in ("index_ms", "index_cpu_ms", "map_cpu_ms", "prefault_ms", "route_ms"):
            phases.setdefault("wt_open_" + k, []).append(ot[k])
        phases["files_mapped"] = ot["files_mapped"]
        phases["files_registered"] = ot["files_registered"]
    if trace is not None:
        recs = h.trace(origin.cuda_event)
        batch_of = {r["event"]: r["index"] for r in recs if r["kind"] == "ingest"}
        for r in recs:
            if r["kind"] == "gemv":
                r["batch"] = batch_of.get(r["event"])
        for r in recs:
            r.pop("event", None)
        trace.append({"records": recs, "host_ms": dt * 1e3, "open_ms": (t1 - t0) * 1e3,
                      "alloc_ms": (ta - t1) * 1e3})
    launches = h.kernel_launches()
    status = h.device_status()
    h.close()
    if slab is None:
        del sl, dev
    return dt, launches, status, len(mats)


def evict_page_cache(paths):
    """Drop the files' pages from the page cache (posix_fadvise DONTNEED on each file only)."""
    for p in paths:
        fd = os.open(p, os.O_RDONLY)
        try:
            os.fdatasync(fd)
            os.posix_fadvise(fd, 0, 0, os.POSIX_FADV_DONTNEED)
        finally:
            os.close(fd)


def quartiles(v):
    """(q1, q3) of a sample (inclusive method; the sample itself when shorter than 2)."""
    if len(v) < 2:
        return (v[0], v[0]) if v else (float("nan"), float("nan"))
    q = statistics.quantiles(v, n=4, method="inclusive")
    return q[0], q[2]


def run_wt(args, rank, world):
    ck, gen_s = make_files(args, rank, world)
    import torch
    from paper_2608_12114_gb300 import build, pipeline, wt

    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
        dist.barrier()
    if rank == 0:
        build.build()
    if dist:
        dist.barrier()
    build.build()  # no-op when fresh; loads the same in-tree library on every rank
    mode = {"gather": wt.WT_ADOPT_GATHER, "ce": wt.WT_ADOPT_CE, "staged": wt.WT_ADOPT_STAGED}[args.mode]
    oflags = open_flags(wt, args.open)

    probe = h2d_probe(torch)
    h2d = max(probe.values())
    log("H2D ceilings %s GB/s; files %.2f GB generated in %.1f s" % (probe, ck.data_bytes / 1e9, gen_s))

    # buffers for the resident pass and the no-allocation first-use variant (allocated once)
    h0 = wt.Handle(ck.paths)
    mats = pipeline.matrices(h0)
    x_host = pipeline.host_inputs(mats)  # the step's inputs, pinned: copied in every timed run
    slab = make_slab(torch, pipeline, h0, mats, x_host=x_host)
    dev, xs, ys = slab["dev"], slab["xs"], slab["ys"]
    rows = [mats[k].shape[0] for k in dev.gemv_mats()]
    y_host = torch.empty(sum(rows), dtype=torch.float32, pin_memory=True)  # host copy of every y
    weight_bytes = dev.weight_bytes
    data_bytes = ck.data_bytes
    gdt = {dev.mats[k].dtype for k in dev.gemv_mats()}
    alg_bytes = sum(gemv_alg_bytes(dev.mats[k].dtype, *dev.mats[k].shape) for k in dev.gemv_mats()) \
        if len(gdt) == 1 else None
    wdt = DT_NAME[gdt.pop()] if len(gdt) == 1 else "mixed"
    torch.cuda.synchronize()

    ingest_s, consume_s = torch.cuda.Stream(), consumer_stream(torch, args)

    # ---------------- e2e: file -> first use (1 warm-up, then timed repetitions), with the
    # device buffers allocated inside each run (fresh), and with buffers allocated once (reused)
    def e2e_series(fresh):
        times, launches, ph = [], 0, {}
        for rep in range(0 if args.skip_e2e else 1 + args.e2e_reps):
            if dist:
                dist.barrier()
            dt, nl, st, nm = first_use(torch, wt, pipeline, ck, mode, ingest_s, consume_s, x_host, y_host,
                                       None if fresh else slab, ph if rep > 0 else None, flags=oflags)
            if st != 0:
                raise SystemExit("device status %d after first-use run" % st)
            if rep > 0:
                times.append(dt)
                launches = nl
        return times, launches, ph

    if not args.skip_e2e:
        del slab["dev"], slab["ys"], slab["yflat"], slab["xdev"]  # the reused buffers go back while fresh runs allocate
        dev = ys = None
        torch.cuda.empty_cache()
    e2e_times, e2e_launches, phases = e2e_series(True)
    if not args.skip_e2e:
        slab = make_slab(torch, pipeline, h0, mats, x_host=x_host)
        dev, xs, ys = slab["dev"], slab["xs"], slab["ys"]
    reuse_times, _, reuse_phases = e2e_series(False)
    e2e_s = statistics.median(e2e_times) if e2e_times else float("nan")
    e2e_gbs = data_bytes / e2e_s / 1e9
    reuse_s = statistics.median(reuse_times) if reuse_times else float("nan")
    log("file->first-use with allocation: %.1f ms median (%s), %.1f GB/s = %.1f%% of the H2D ceiling; "
        "buffers reused: %.1f ms, %.1f GB/s" % (
            e2e_s * 1e3, ", ".join("%.1f" % (t * 1e3) for t in e2e_times), e2e_gbs, 100 * e2e_gbs / h2d,
            reuse_s * 1e3, data_bytes / reuse_s / 1e9))

    cold = None
    if args.cold_reps and not args.skip_e2e:
        # storage-bound variant (the precondition of Algorithm 2 fails): the files' pages are
        # evicted before each run; reported apart from the warm-cache headline
        ct = []
        for _ in range(args.cold_reps):
            evict_page_cache(ck.paths)
            ct.append(first_use(torch, wt, pipeline, ck, mode, ingest_s, consume_s, x_host, y_host, slab)[0])
        cold = {"value": round(aggregate_gbs(data_bytes, world, statistics.median(ct)), 1), "unit": "GB/s",
                "ms": [round(t * 1e3, 1) for t in ct],
                "what": "file -> first use after posix_fadvise(DONTNEED) on the checkpoint files: storage-bound"}
        log("cold file->first-use: %s ms" % cold["ms"])

    arms = {}
    if args.arms:
        # the mode order rotates across repetitions so no arm always runs first
        names = [("gather", wt.WT_ADOPT_GATHER), ("ce", wt.WT_ADOPT_CE), ("staged", wt.WT_ADOPT_STAGED), ("stock_torch", None)]
        ts = {n: [] for n, _ in names}
        for r in range(3):
            for n, m in names[r:] + names[:r]:
                if m is None:
                    ts[n].append(data_bytes / stock_torch_arm(torch, ck, wt, pipeline))
                else:
                    ts[n].append(first_use(torch, wt, pipeline, ck, m, ingest_s, consume_s, x_host, y_host, slab)[0])
        arms = {n: round(data_bytes / statistics.median(v) / 1e9, 1) for n, v in ts.items()}
        log("ingest arms GB/s (median of 3, rotated order):", arms)

    h0.close()

    # ---------------- resident pass: the steady-state consumer
    h = wt.Handle(ck.paths, oflags)
    ev = dev.adopt(h, mode, ingest_s.cuda_stream)
    ingest_s.synchronize()
    descs = dev.descs(xs, ys)
    s = consume_s
    for _ in range(args.warmup):
        h.pass_(descs, s.cuda_stream)
    s.synchronize()
    graph, graph_launches = None, 0
    gp = max(1, args.graph_passes) if args.graph else 1
    if gp > 1:
        args.steps = -(-args.steps // gp) * gp
    if args.graph:
        # gp resident passes captured into one CUDA graph; each replay runs gp steps with no
        # host work between them (the replay's own launch is paid once per gp passes)
        n_cap = h.kernel_launches()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=s):
            for _ in range(gp):
                h.pass_(descs, torch.cuda.current_stream().cuda_stream)
        graph_launches = (h.kernel_launches() - n_cap) / gp
        with torch.cuda.stream(s):
            for _ in range(args.warmup):
                graph.replay()
        s.synchronize()
    n0 = h.kernel_launches()
    nrec = args.steps // gp
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(nrec + 1)]
    if dist:
        dist.barrier()
    torch.cuda.synchronize()
    with Clocks(bus_id()) as clk:
        evs[0].record(s)
        if graph is not None:
            with torch.cuda.stream(s):
                for i in range(nrec):
                    graph.replay()
                    evs[i + 1].record(s)
        else:
            for i in range(args.steps):
                h.pass_(descs, s.cuda_stream)
                evs[i + 1].record(s)
        s.synchronize()
    torch.cuda.synchronize()
    if dist:
        dist.barrier()
    launches = int(round(h.kernel_launches() - n0 + graph_launches * args.steps))
    per = [evs[i].elapsed_time(evs[i + 1]) / gp for i in range(nrec)]
    total_ms = evs[0].elapsed_time(evs[-1])
    status = h.device_status()
    h.close()
    stamps = run_stamps(torch, wt, descs, s, args, gp) if args.stamps and status == 0 else None
    if status != 0:
        raise SystemExit("device status %d after resident passes" % status)

    total_ms, e2e_s_max = combine_ranks(dist, "cuda", total_ms, e2e_s)
    ms_per_step = total_ms / args.steps
    value = aggregate_gbs(weight_bytes * args.steps, world, total_ms / 1e3)
    launches_per_pass = launches / args.steps
    avg_launch_ms = statistics.mean(per) if launches_per_pass == 1 else None
    peak, peak_kind = measured_peaks()
    roof = None
    if avg_launch_ms and alg_bytes:
        achieved = alg_bytes / (avg_launch_ms / 1e3) / 1e9
        tr = kernel_traffic("gemv_tma_large_traffic.json") if args.workload == "large" else None
        roof = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                "frac": round(achieved / peak, 4), "peak_kind": peak_kind,
                "traffic": (tr["dram_bytes_per_launch_full"] if tr else None),
                "algorithmic_bytes_per_launch": alg_bytes,
                "kernel": onecol_kernel_name(wdt, [dev.mats[k].shape for k in dev.gemv_mats()]),
                "frac_of_nominal_8TBps": round(achieved / NOMINAL_HBM_GBS, 4)}
    clocks = clk.summary()
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": wdt,
        "data": DATA_DESC.get(wdt, "synthetic"),
        "config": {"workload": workload_desc(args), "weight_bytes": weight_bytes, "data_bytes": data_bytes,
                   "files": len(ck.paths), "matrices": len(dev.gemv_mats()), "ingest_mode": args.mode,
                   "consumer_stream_priority": args.consumer_priority,
                   "open": {"map": "mapped", "nomap": "WT_OPEN_NOMAP (pread)", "prefault": "mapped, WT_OPEN_PREFAULT",
                            "register": "mapped, WT_ROUTE_REGISTER",
                            "maplarge": "WT_OPEN_MAP_LARGE: files of >= %s bytes mapped, smaller ones read with pread"
                                        % os.environ.get("WT_MAP_MIN_BYTES", wt.WT_MAP_MIN_BYTES)}[args.open],
                   "l2": ("inputs larger than L2 (no flush)" if weight_bytes > L2_BYTES else
                          "inputs smaller than L2, no flush: passes may hit L2 (a dispatch-overhead point)"),
                   "parallelism": "replicas" if world > 1 else "1 GPU",
                   "cuda_graph": bool(args.graph), "passes_per_graph": gp if args.graph else None},
        "resident_frac_of_hbm": {"measured": round(value / world / peak, 4), "nominal_8TBps": round(value / world / NOMINAL_HBM_GBS, 4)},
        "clocks": clocks,
        "e2e": {"value": round(aggregate_gbs(data_bytes, world, e2e_s_max), 1), "unit": "GB/s",
                "h2d_bytes_per_step": data_bytes + int(x_host.numel()), "d2h_bytes_per_step": int(y_host.numel() * 4),
                "ms": round(e2e_s * 1e3, 2), "pinned_h2d_gbs": round(h2d, 1), "h2d_ceilings_gbs": probe,
                "frac_of_pinned_h2d": round(e2e_gbs / h2d, 4), "reps": args.e2e_reps,
                "what": "wt_open + device allocation of the slabs, x and y (fresh each run, after "
                        "torch.cuda.empty_cache; slabs allocated segment by segment between wt_adopt "
                        "calls, x and y in the first one) + wt_adopt + H2D of every x from pinned host "
                        "memory + event-gated first pass + D2H of all y, page cache warm; the library's "
                        "own status word and plan tables come from its per-device block cache; "
                        "pinned_h2d_gbs is the highest of h2d_ceilings_gbs; phases: alloc_ms is host "
                        "time in allocations, enqueue_ms the rest of the time to the last return; "
                        "wt_open_*: wt_open's own step times (wt_open_times: parallel index + map loop, "
                        "summed per-file index and mmap time, prefault, route probe)",
                "launches_per_run": e2e_launches,
                "iqr_ms": [round(v * 1e3, 2) for v in quartiles(e2e_times)] if e2e_times else None,
                "phases_ms_median": {k: round(statistics.median(v), 2) for k, v in phases.items() if k.endswith("_ms")},
                "route": phases.get("route"),
                "files_mapped": phases.get("files_mapped"), "files_registered": phases.get("files_registered"),
                "buffers_reused": {"value": round(aggregate_gbs(data_bytes, world, reuse_s), 1), "unit": "GB/s",
                                   "ms": round(reuse_s * 1e3, 2),
                                   "frac_of_pinned_h2d": round(data_bytes / reuse_s / 1e9 / h2d, 4),
                                   "phases_ms_median": {k: round(statistics.median(v), 2)
                                                        for k, v in reuse_phases.items() if k.endswith("_ms")},
                                   "what": "the same run with the device buffers allocated once, before it"}},
        "gpu_launches": int(launches),
        "roofline": roof,
    }
    if stamps:
        out["stamps"] = stamps
    if arms:
        out["ingest_arms_gbs"] = arms
    if cold:
        out["e2e_cold"] = cold
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(args, ck, args.cpu_seconds)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if dist:
        dist.barrier()
        dist.destroy_process_group()


def stock_torch_arm(torch, ck, wt, pipeline):
    """The stock path: file bytes -> CPU tensor -> .to('cuda') per tensor, then F.linear."""
    import numpy as np
    h = wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    total = 0
    for f, p in enumerate(ck.paths):
        mm = np.memmap(p, dtype=np.uint8, mode="r")
        for t in h.tensors:
            if t.file != f:
                continue
            cpu = torch.from_numpy(np.array(mm[t.offset:t.offset + t.nbytes]))
            g = cpu.to("cuda")
            if len(t.shape) == 2 and t.dtype == wt.WT_BF16:
                W = g.view(torch.bfloat16).view(t.shape)
                x = torch.ones(t.shape[1], dtype=torch.bfloat16, device="cuda")
                torch.nn.functional.linear(x, W)
            total += t.nbytes
        del mm
    torch.cuda.synchronize()
    h.close()
    return total / (time.perf_counter() - t0)


# ----------------------------------------------------------------------------- the oracle (CPU)

class OracleSample:
    """The oracle, as it stands, walking the workload's matrices in layer order in row blocks.

    Files are parsed (read in full, index decoded) when the walk first reaches them; every
    block is an fp64 GEMV of up to 1024 rows.  run(budget) stops after `budget_s` of work."""

    BLOCK = 1024

    def __init__(self, ck):
        import oracle
        oracle.build()
        self.oracle = oracle
        self.ck = ck
        self.files = {}
        self.parse_s = 0.0
        self.parsed = 0
        self.m = 0
        self.r = 0
        self.xs = {}

    def _blob(self, i):
        t = self.ck.tensors[i]
        if t.file not in self.files:
            t0 = time.perf_counter()
            fo = self.oracle.load(self.ck.paths[t.file])
            self.parse_s += time.perf_counter() - t0
            self.parsed += fo.size
            self.files[t.file] = (fo, {e["name"]: k for k, e in enumerate(fo.entries)})
        fo, names = self.files[t.file]
        return fo.blob(names[t.name])

    def run(self, budget_s):
        """GEMV row blocks until the budget is spent; returns (weight bytes, GEMV seconds)."""
        import numpy as np
        from paper_2608_12114_gb300 import synth
        done_b, gemv_s = 0, 0.0
        t_end = time.perf_counter() + budget_s
        while time.perf_counter() < t_end:
            m = self.ck.matrices[self.m]
            blobs = [self._blob(i) for i in m.parts]
            W = blobs[0] if len(blobs) == 1 else np.concatenate(blobs)
            key = (m.K, m.dtype)
            if key not in self.xs:
                self.xs[key] = synth.make_x(m.K, m.dtype)
            r1 = min(m.M, self.r + self.BLOCK)
            t0 = time.perf_counter()
            self.oracle.gemv_rows(W, m.dtype, m.M, m.K, self.xs[key], range(self.r, r1))
            gemv_s += time.perf_counter() - t0
            done_b += (r1 - self.r) * m.K * synth.ELEM_SIZE[m.dtype]
            self.r = r1
            if self.r == m.M:
                self.m, self.r = (self.m + 1) % len(self.ck.matrices), 0
        return done_b, gemv_s

    def close(self):
        for fo, _ in self.files.values():
            fo.close()
        self.files = {}

    def describe(self, wbytes):
        return ("oracle walk over the workload's matrices in layer order, %.2f GB of weights in "
                "1024-row blocks (%d of %d files parsed, %.2f GB read at %.2f GB/s)" % (
                    wbytes / 1e9, len(self.files), len(self.ck.paths), self.parsed / 1e9,
                    self.parsed / self.parse_s / 1e9 if self.parse_s else 0.0))


def cpu_baseline(args, ck, budget_s):
    """The oracle on the host cores over a bounded sample (about `budget_s` of CPU work)."""
    o = OracleSample(ck)
    wb, gs = o.run(budget_s)
    desc = o.describe(wb)
    parse_rate = o.parsed / o.parse_s if o.parse_s else None
    o.close()
    gemv_rate = wb / gs if gs else None
    first = (1.0 / (1.0 / parse_rate + 1.0 / gemv_rate)) if parse_rate and gemv_rate else None
    return {"value": round(gemv_rate / 1e9, 4) if gemv_rate else None, "unit": "GB/s", "cores": 1,
            "kind": "oracle", "sample": desc + "; value = fp64 GEMV weight GB/s",
            "cores_available": len(os.sched_getaffinity(0)),
            "parse_gbs": round(parse_rate / 1e9, 3) if parse_rate else None,
            "first_use_gbs": round(first / 1e9, 4) if first else None}


def run_reference(args, rank, world):
    """The reference arm: the CPU oracle as it stands, on the same workload, metric and unit.
    Each step is a bounded slice of the oracle's walk; the run stays within a few minutes."""
    if rank != 0:
        return
    ck, gen_s = make_files(args, 0, 1)
    steps, warm = max(1, args.steps), max(0, args.warmup)
    budget = min(10.0, max(0.05, args.ref_seconds / (steps + warm)))
    o = OracleSample(ck)
    rates, tot_b, tot_s = [], 0, 0.0
    for i in range(warm + steps):
        wb, gs = o.run(budget)
        if i >= warm and gs > 0:
            rates.append(wb / gs)
            tot_b += wb
            tot_s += gs
    desc = o.describe(tot_b)
    parse_rate = o.parsed / o.parse_s if o.parse_s else None
    o.close()
    v = statistics.median(rates) / 1e9
    first = 1.0 / (1.0 / parse_rate + 1.0 / (tot_b / tot_s)) / 1e9 if parse_rate else None
    cb = {"value": round(v, 4), "unit": "GB/s", "cores": 1, "kind": "oracle",
          "sample": "%d steps of %.2f s each: %s" % (steps, budget, desc)}
    out = {"impl": "reference", "metric": METRIC, "value": round(v, 4), "unit": "GB/s", "n_gpus": 1,
           "steps": steps, "warmup": warm, "ms_per_step": round(tot_s / max(1, len(rates)) * 1e3, 2),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": {"workload": workload_desc(args)}, "cpu_baseline": cb,
           "e2e": {"value": round(first, 4) if first else None, "unit": "GB/s",
                   "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0,
                   "what": "1 / (1/parse GB/s + 1/GEMV GB/s) of the oracle"}}
    print(json.dumps(out), flush=True)


def overlap_summary(recs):
    """Contract C3 read off one traced first use: when each GEMV group ran against the batch it
    waited on, the tail after the last batch, and the serial time it would take otherwise."""
    ing = [r for r in recs if r["kind"] == "ingest"]
    gem = [r for r in recs if r["kind"] == "gemv"]
    if not ing or not gem:
        return {}
    end_of = {r["index"]: r["end_ms"] for r in ing}
    last_ing = max(r["end_ms"] for r in ing)
    first_ing = min(r["begin_ms"] for r in ing)
    lags = [g["begin_ms"] - end_of[g["batch"]] for g in gem if g.get("batch") in end_of]
    busy = sum(g["end_ms"] - g["begin_ms"] for g in gem)
    before = sum(max(0.0, min(g["end_ms"], last_ing) - g["begin_ms"]) for g in gem)
    # a group finished before the next batch landed: it did not wait for a full drain
    nxt = sorted(end_of.items())
    early = 0
    for g in gem:
        b = g.get("batch")
        later = [e for i, e in nxt if b is not None and i > b]
        if later and g["end_ms"] <= later[0]:
            early += 1
    # time the link had nothing queued: gaps between one batch landing and the next beginning
    order = sorted(ing, key=lambda r: r["begin_ms"])
    idle = sum(max(0.0, b["begin_ms"] - a["end_ms"]) for a, b in zip(order, order[1:]))
    return {"batches": len(ing), "groups": len(gem),
            "first_batch_begin_ms": round(first_ing, 3),
            "link_idle_ms": round(idle, 3),
            "ingest_span_ms": round(last_ing - first_ing, 3),
            "ingest_gbs": round(sum(r["bytes"] for r in ing) / (last_ing - first_ing) / 1e6, 1),
            "gemv_busy_ms": round(busy, 3),
            "gemv_busy_before_last_batch_ms": round(before, 3),
            "groups_done_before_next_batch": early,
            "lag_ms_median": round(statistics.median(lags), 4) if lags else None,
            "lag_ms_max": round(max(lags), 4) if lags else None,
            "tail_ms": round(max(g["end_ms"] for g in gem) - last_ing, 4),
            "first_use_device_ms": round(max(g["end_ms"] for g in gem) - first_ing, 3),
            "serial_estimate_ms": round(last_ing - first_ing + busy, 3)}


def run_timeline(args):
    """One file -> first-use run traced on the device (WT_OPEN_TIMELINE): per ingest batch its
    begin/end, per GEMV group its begin/end and the batch it waited on."""
    ck, gen_s = make_files(args, 0, 1)
    import torch
    from paper_2608_12114_gb300 import build, pipeline, wt
    build.build()
    torch.cuda.set_device(0)
    mode = {"gather": wt.WT_ADOPT_GATHER, "ce": wt.WT_ADOPT_CE, "staged": wt.WT_ADOPT_STAGED}[args.mode]
    oflags = open_flags(wt, args.open)
    h0 = wt.Handle(ck.paths, oflags)
    mats = pipeline.matrices(h0)
    x_host = pipeline.host_inputs(mats)
    slab = make_slab(torch, pipeline, h0, mats, x_host=x_host)
    rows = sum(mats[k].shape[0] for k in slab["dev"].gemv_mats())
    y_host = torch.empty(rows, dtype=torch.float32, pin_memory=True)
    ingest_s, consume_s = torch.cuda.Stream(), consumer_stream(torch, args)
    if args.fresh:  # every run allocates its own buffers; this one goes back first
        del slab["dev"], slab["ys"], slab["yflat"], slab["xdev"]
        slab = None
    for _ in range(2):  # warm-up, untraced
        first_use(torch, wt, pipeline, ck, mode, ingest_s, consume_s, x_host, y_host, slab, flags=oflags)
    runs = []
    for _ in range(max(1, min(args.e2e_reps, 5))):
        tr = []
        first_use(torch, wt, pipeline, ck, mode, ingest_s, consume_s, x_host, y_host, slab, flags=oflags, trace=tr)
        runs.append(tr[0])
    h0.close()
    sums = [overlap_summary(r["records"]) for r in runs]
    best = min(range(len(runs)), key=lambda i: runs[i]["host_ms"])
    out = {"metric": "first-use overlap timeline (ingest batches vs event-gated GEMV groups)",
           "config": {"workload": workload_desc(args), "ingest_mode": args.mode,
                      "data_bytes": ck.data_bytes, "runs": len(runs),
                      "buffers": "allocated inside each run" if args.fresh else "allocated once, reused"},
           "summaries": sums, "host_ms": [round(r["host_ms"], 3) for r in runs],
           "open_ms": [round(r["open_ms"], 3) for r in runs], "alloc_ms": [round(r["alloc_ms"], 3) for r in runs],
           "records": runs[best]["records"]}
    log("timeline:", json.dumps(sums[best]))
    print(json.dumps(out), flush=True)


def run_cube(args):
    """Table "cube" and the ordering figure (Sec. 4) on this GPU, protocol workload by default."""
    if args.workload == "large":
        args.workload = "protocol"
    ck, gen_s = make_files(args, 0, 1)
    import torch
    from paper_2608_12114_gb300 import build, contract
    build.build()
    torch.cuda.set_device(0)
    out = contract.measure(ck.paths, reps=max(3, min(args.e2e_reps, 9)))
    out.update({"metric": "execution-contract ablation: idle GB/s per cell, excess ms per pass over an "
                          "in-flight framework workload", "config": {"workload": workload_desc(args)},
                "cells": "(weights, activations, ordering): map = C1 on, device = C2 on, stream = C3 on"})
    print(json.dumps(out), flush=True)


def run_policy(args):
    """Algorithm 2 (Sec. 8.1) on this GPU for the workload: a GB300 row of Table "policy"."""
    ck, gen_s = make_files(args, 0, 1)
    import torch
    from paper_2608_12114_gb300 import build, policy
    build.build()
    torch.cuda.set_device(0)
    h2d = pinned_h2d_gbs(torch)
    out = policy.measure_gb300(ck.paths, reps=max(3, min(args.e2e_reps, 9)))
    d = out.as_dict()
    d.update({"metric": "endpoint selection (Algorithm 2): W/B per endpoint", "unit": "ms",
              "config": {"workload": workload_desc(args)}, "pinned_h2d_gbs": round(h2d, 1),
              "what": "map = GEMV reads the prefaulted file mapping in place; resident = GEMV over an HBM "
                      "copy; copy = wt_adopt into HBM then the event-gated GEMV, every pass"})
    print(json.dumps(d), flush=True)


def run_tsweep(args):
    """The T-sweep (Sec. 4.3): one multi-column pass over every matrix with T activation
    columns, resident in HBM (CUDA events over `steps` passes), per-use copy (wt_adopt + the
    event-gated pass, wall time per rep), and the map endpoint (W read in place from the
    file mapping: the paper's adoption arm; CUDA events)."""
    if args.workload == "large":
        args.workload = "protocol_q8"
    ts = [int(v) for v in args.tsweep.split(",")]
    ck, gen_s = make_files(args, 0, 1)
    import torch
    from paper_2608_12114_gb300 import build, pipeline, wt
    build.build()
    torch.cuda.set_device(0)
    h = wt.Handle(ck.paths)
    mats = pipeline.matrices(h)
    dev = pipeline.DeviceCheckpoint.allocate(h, mats)
    ks = dev.gemv_mats()
    s = torch.cuda.Stream()
    ingest = torch.cuda.Stream()
    dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
    s.synchronize()
    wbytes = dev.weight_bytes
    peak, peak_kind = measured_peaks()
    g = torch.Generator(device="cpu").manual_seed(1234)
    rows = []
    with Clocks(bus_id()) as clk:
        for T in ts:
            n = max(T, 1)
            xs = {}
            for k in ks:
                m = dev.mats[k]
                key = (m.shape[1], m.dtype)
                if key not in xs:
                    xdt = torch.bfloat16 if m.dtype == wt.WT_BF16 else torch.float16
                    xs[key] = torch.randn(n, m.shape[1], generator=g).to(xdt).cuda()
            ys = {k: torch.empty(n * dev.mats[k].shape[0], dtype=torch.float32, device="cuda") for k in ks}
            d = dev.descs(xs, ys)
            d["cols"] = T
            for _ in range(args.warmup):
                h.pass_(d, s.cuda_stream)
            s.synchronize()
            n0 = h.kernel_launches()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(s)
            for _ in range(args.steps):
                h.pass_(d, s.cuda_stream)
            e1.record(s)
            s.synchronize()
            ms = e0.elapsed_time(e1) / args.steps
            launches = (h.kernel_launches() - n0) / args.steps
            if h.device_status() != 0:
                raise SystemExit("device status %d in the T-sweep" % h.device_status())
            copy_ms = []
            for rep in range(max(2, args.e2e_reps) + 1):
                torch.cuda.synchronize()
                t0 = time.perf_counter()
                evs = dev.adopt(h, wt.WT_ADOPT_GATHER, ingest.cuda_stream)
                dc = dev.descs(xs, ys, evs)
                dc["cols"] = T
                h.pass_(dc, s.cuda_stream)
                s.synchronize()
                ingest.synchronize()
                if rep:
                    copy_ms.append((time.perf_counter() - t0) * 1e3)
            cm = statistics.median(copy_ms)
            # map endpoint: W read in place from the file mapping (prefaulted at plan build)
            dm = dev.descs(xs, ys)
            dm["cols"] = T
            dm["W"] = [h.tensors[dev.mats[k].parts[0]].host_ptr for k in ks]
            map_ms = None
            if all(len(dev.mats[k].parts) == 1 for k in ks):
                h.pass_(dm, s.cuda_stream)
                s.synchronize()
                em0, em1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                nmap = max(3, args.steps // 20)
                em0.record(s)
                for _ in range(nmap):
                    h.pass_(dm, s.cuda_stream)
                em1.record(s)
                s.synchronize()
                map_ms = em0.elapsed_time(em1) / nmap
            flops = 2.0 * sum(dev.mats[k].shape[0] * dev.mats[k].shape[1] for k in ks) * n
            two_byte = all(dev.mats[k].dtype in (wt.WT_BF16, wt.WT_F16) for k in ks)
            force = os.environ.get("WT_COLS_KERNEL")
            on_umma = two_byte and (force == "umma" or (force != "mma" and T > 8))
            shapes = [dev.mats[k].shape for k in ks]
            int8 = all(dev.mats[k].dtype == wt.WT_I8 for k in ks)
            kname = (onecol_kernel_name(DT_NAME[dev.mats[ks[0]].dtype], shapes) if T == 0 else
                     "gemm_cols_umma (tcgen05, M128 N16 K16)" if on_umma else
                     int8_tc_kernel(shapes, T) if int8 else "gemm_cols (mma.sync m16n8k16)")
            rows.append({"T": T, "kernel": kname,
                         "ms": round(ms, 4), "weight_gbs": round(wbytes / ms / 1e6, 1),
                         "logical_gbs": round(n * wbytes / ms / 1e6, 1), "tflops": round(flops / ms / 1e9, 2),
                         "frac_of_hbm": round(wbytes / ms / 1e6 / peak, 4), "launches_per_pass": launches,
                         "copy_ms": round(cm, 3), "resident_over_copy": round(cm / ms, 2),
                         "map_ms": round(map_ms, 3) if map_ms else None,
                         "map_over_copy": round(cm / map_ms, 3) if map_ms else None})
            log("T=%d: %.4f ms, %.1f GB/s weights (%.1f%% of %s HBM), copy %.3f ms, map %s ms" % (
                T, ms, wbytes / ms / 1e6, 100 * wbytes / ms / 1e6 / peak, peak_kind, cm,
                "%.3f" % map_ms if map_ms else "-"))
    h.close()
    out = {"metric": "multi-column T-sweep: resident pass time and weight GB/s per T", "unit": "GB/s",
           "config": {"workload": workload_desc(args), "weight_bytes": wbytes, "matrices": len(ks),
                      "steps": args.steps, "warmup": args.warmup, "l2": "inputs larger than L2 (no flush)"},
           "peak_hbm_gbs": peak, "peak_kind": peak_kind, "tsweep": rows, "clocks": clk.summary()}
    print(json.dumps(out), flush=True)


# Issue peak of the SMs: 152 SMs x 4 schedulers x one warp instruction (32 lanes) per clock.
# FNV-1a-64 is integer ALU work, so its ceiling is this rate divided by the instructions the
# kernel spends per byte (ncu's smsp__inst_executed x 32 / bytes), or HBM, whichever is lower.
def issue_peak_lane_ops(sm_mhz, sms=152):
    return sms * 4 * 32 * sm_mhz * 1e6


def run_checksum(args):
    """Step 9 measured: wt_checksum (per-tensor FNV-1a-64 leaf digests plus the combine pass)
    over every tensor of the workload, resident in HBM, CUDA events over `steps` calls on the
    launching stream.  Digests are verification: this is their throughput, outside the
    first-use and resident-pass figures."""
    ck, gen_s = make_files(args, 0, 1)
    import torch
    from paper_2608_12114_gb300 import build, pipeline, wt
    build.build()
    torch.cuda.set_device(0)
    h = wt.Handle(ck.paths)
    mats = pipeline.matrices(h)
    dev = pipeline.DeviceCheckpoint.allocate(h, mats)
    s = torch.cuda.Stream()
    dev.adopt(h, wt.WT_ADOPT_GATHER, s.cuda_stream)
    s.synchronize()
    idx = sorted(dev.dst)
    ptrs = [dev.dst[i] for i in idx]
    nb = [h.tensors[i].nbytes for i in idx]
    total = sum(nb)
    out = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
    base = out.data_ptr()
    outs = [base + 8 * j for j in range(len(idx))]

    def call():
        h.checksum(ptrs, nb, base, s.cuda_stream)

    for _ in range(max(3, args.warmup)):
        call()
    s.synchronize()
    first = out.clone()
    steps = max(1, min(args.steps, 50))
    n0 = h.kernel_launches()
    with Clocks(bus_id()) as clk:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(s)
        for _ in range(steps):
            call()
        e1.record(s)
        s.synchronize()
    ms = e0.elapsed_time(e1) / steps
    launches = (h.kernel_launches() - n0) / steps
    stable = bool(torch.equal(first, out))
    h.close()
    peak, peak_kind = measured_peaks()
    gbs = total / ms / 1e6
    csum = clk.summary()
    row = {"metric": "per-tensor FNV-1a-64 digest throughput (wt_checksum, leaf tree)", "value": round(gbs, 1),
           "unit": "GB/s", "ms_per_call": round(ms, 4), "bytes_per_call": total, "tensors": len(idx),
           "launches_per_call": launches, "digests_repeat": stable, "frac_of_hbm": round(gbs / peak, 4),
           "peak_hbm_gbs": peak, "peak_kind": peak_kind,
           "issue_peak_lane_ops_per_s": issue_peak_lane_ops(csum.get("sm_mhz") or 2070.0),
           "config": {"workload": workload_desc(args), "steps": steps, "l2": "inputs larger than L2 (no flush)"
                      if total > L2_BYTES else "inputs smaller than L2"},
           "clocks": csum}
    log("checksum: %.4f ms per call, %.1f GB/s (%.1f%% of %s HBM), %d launches, digests repeat: %s" % (
        ms, gbs, 100 * gbs / peak, peak_kind, launches, stable))
    print(json.dumps(row), flush=True)


def main():
    args = parse_args()
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return
    if args.policy:
        run_policy(args)
        return
    if args.timeline:
        run_timeline(args)
        return
    if args.tsweep:
        run_tsweep(args)
        return
    if args.cube:
        run_cube(args)
        return
    if args.checksum:
        run_checksum(args)
        return
    run_wt(args, rank, world)


if __name__ == "__main__":
    main()
