"""The C ABI library loads, exports every entry point of include/wt.h, and its host-side
parser agrees with the oracle (no GPU needed: WT_OPEN_HOST_ONLY makes no CUDA call)."""
import os
import re

import pytest

import oracle
from paper_2608_12114_gb300 import build, synth, wt
from tests import _files

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return wt.lib()


def declared_symbols():
    """Every wt_* function declared in include/*.h."""
    inc = os.path.join(ROOT, "include")
    src = "".join(open(os.path.join(inc, f)).read() for f in sorted(os.listdir(inc)) if f.endswith(".h"))
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(wt_[a-z_]+)\s*\(", src)))


def test_every_declared_symbol_is_exported(L):
    decl = declared_symbols()
    assert len(decl) >= 15
    for s in decl:
        assert hasattr(L, s), s
    assert sorted(wt.SYMBOLS) == decl
    assert L.wt_abi_version() == 4


def test_only_the_abi_is_exported(L):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", wt.LIB_PATH], capture_output=True, text=True).stdout
    exported = sorted({l.split()[-1] for l in out.splitlines() if " T " in l})
    assert exported == declared_symbols()


def test_host_only_parse_matches_oracle(L, tmp_path):
    ck = synth.build("mid", str(tmp_path / "mid"), layers=2, vocab=96)
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
        assert h.n_files == len(ck.paths)
        got = [(t.name, t.dtype, t.shape, t.nbytes, t.file, t.offset) for t in h.tensors]
        want = []
        for f, p in enumerate(ck.paths):
            for e in oracle.load(p).entries:
                want.append((e["name"], e["dtype"], e["shape"], e["nbytes"], f, e["offset"]))
        assert got == want
        assert all(h.route(f) == wt.WT_ROUTE_NONE for f in range(h.n_files))
        assert h.find("layers.1.down") == [t.name for t in h.tensors].index("layers.1.down")
        with pytest.raises(wt.WtError) as ei:
            h.find("nope")
        assert ei.value.code == wt.WT_EINVAL


def test_host_ptr_points_at_file_bytes(L, tmp_path):
    import ctypes
    ck = synth.build("tiny", str(tmp_path))
    of = oracle.load(ck.paths[0])
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
        for i, t in enumerate(h.tensors):
            assert ctypes.string_at(t.host_ptr, t.nbytes) == of.blob(i).tobytes()


@pytest.mark.parametrize("label,img", _files.bad_files(), ids=[b[0] for b in _files.bad_files()])
def test_rejections_agree_with_oracle(L, tmp_path, label, img):
    p = str(tmp_path / (label + ".wt"))
    with open(p, "wb") as f:
        f.write(img)
    with pytest.raises(oracle.OracleError):
        oracle.load(p)
    with pytest.raises(wt.WtError) as ei:
        wt.Handle([p], wt.WT_OPEN_HOST_ONLY)
    assert ei.value.code == wt.WT_EFORMAT
    assert p in str(ei.value)


def test_good_hand_built_file(L, tmp_path):
    img, (o1, ba), (o2, bb) = _files.good_two_entry()
    p = str(tmp_path / "g.wt")
    open(p, "wb").write(img)
    with wt.Handle([p], wt.WT_OPEN_HOST_ONLY) as h:
        assert [(t.name, t.shape, t.offset, t.nbytes) for t in h.tensors] == [("a", (2, 4), o1, 16), ("b", (3,), o2, 6)]


def test_missing_file_and_bad_arguments(L, tmp_path):
    with pytest.raises(wt.WtError) as ei:
        wt.Handle([str(tmp_path / "missing.wt")], wt.WT_OPEN_HOST_ONLY)
    assert ei.value.code == wt.WT_EIO
    with pytest.raises(wt.WtError) as ei:
        wt.Handle([], 1 << 12)
    assert ei.value.code == wt.WT_EINVAL


def test_one_bad_file_leaves_nothing_open(L, tmp_path):
    ck = synth.build("many", str(tmp_path / "m"), n_matrices=20)
    bad = str(tmp_path / "bad.wt")
    open(bad, "wb").write(b"WTCKPT02" + b"\0" * 64)
    with pytest.raises(wt.WtError):  # first call starts the library's thread pool
        wt.Handle([bad], wt.WT_OPEN_HOST_ONLY)
    fds0 = len(os.listdir("/proc/self/fd"))
    for _ in range(5):
        with pytest.raises(wt.WtError):
            wt.Handle(ck.paths[:20] + [bad] + ck.paths[20:], wt.WT_OPEN_HOST_ONLY)
    assert len(os.listdir("/proc/self/fd")) == fds0
    assert not [l for l in open("/proc/self/maps") if str(tmp_path) in l]  # no checkpoint stays mapped


def test_open_close_cycles_are_flat(L, tmp_path):
    ck = synth.build("many", str(tmp_path / "c"), n_matrices=10)
    h = wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)
    assert [l for l in open("/proc/self/maps") if str(tmp_path) in l]  # mapped while open
    h.close()
    fds0 = len(os.listdir("/proc/self/fd"))
    for _ in range(200):
        wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()
    assert len(os.listdir("/proc/self/fd")) == fds0
    assert not [l for l in open("/proc/self/maps") if str(tmp_path) in l]


def test_device_calls_refused_on_host_only_handle(L, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
        with pytest.raises(wt.WtError) as ei:
            h.adopt([0], [1 << 20])
        assert ei.value.code == wt.WT_ENOTSUP
        with pytest.raises(wt.WtError) as ei:
            h.pass_([wt.gemv_desc(16, wt.WT_F32, 1, 4, 16, 16)])
        assert ei.value.code == wt.WT_ENOTSUP
        assert h.device_status() == 0


def test_live_counts_follow_handles(L, tmp_path):
    ck = synth.build("many", str(tmp_path / "lv"), n_matrices=4)
    base = wt.live()
    hs = [wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) for _ in range(3)]
    assert wt.live()["handles"] == base["handles"] + 3
    for h in hs:
        h.close()
    assert wt.live() == base
    # a failed open leaves no handle behind
    with pytest.raises(wt.WtError):
        wt.Handle(ck.paths + [str(tmp_path / "missing.wt")], wt.WT_OPEN_HOST_ONLY)
    assert wt.live() == base


def test_registration_and_trace_queries_on_host_only_handle(L, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
        assert h.registration(0) == 0  # nothing is registered without a device route
        with pytest.raises(wt.WtError) as ei:
            h.registration(1)
        assert ei.value.code == wt.WT_EINVAL
        with pytest.raises(wt.WtError) as ei:  # no timeline: the handle was not opened with one
            h.trace(1)
        assert ei.value.code == wt.WT_EINVAL
    # TIMELINE is a known flag (a host-only handle ignores it)
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_TIMELINE).close()


def header_defines():
    """Every integer #define of include/wt.h: name -> value."""
    src = open(os.path.join(ROOT, "include", "wt.h")).read()
    return {m.group(1): int(m.group(2)) << int(m.group(3) or 0)
            for m in re.finditer(r"#define\s+(WT_[A-Z0-9_]+)\s+\(?([0-9]+)u?(?:\s*<<\s*([0-9]+))?\)?", src)}


def test_binding_constants_match_the_header():
    d = header_defines()
    for name in ("WT_OPEN_HOST_ONLY", "WT_OPEN_PREFAULT", "WT_OPEN_TIMELINE", "WT_OPEN_NOMAP", "WT_OPEN_STAMPS",
                 "WT_OPEN_MAP_LARGE", "WT_MAP_MIN_BYTES",
                 "WT_TRACE_INGEST", "WT_TRACE_GEMV", "WT_ADOPT_GATHER", "WT_ADOPT_CE", "WT_ADOPT_STAGED"):
        assert d[name] == getattr(wt, name), name
    # the stamp record: field order and width
    assert d["WT_STAMP_FIELDS"] == len(wt.STAMP_FIELDS)
    for i, f in enumerate(wt.STAMP_FIELDS):
        assert d["WT_STAMP_" + f.upper()] == i, f


def test_map_large_maps_only_the_large_files(L, tmp_path, monkeypatch):
    ck = synth.build("many", str(tmp_path / "ml"), n_matrices=40)
    sizes = [os.path.getsize(p) for p in ck.paths]
    thr = sorted(sizes)[len(sizes) // 2]
    monkeypatch.setenv("WT_MAP_MIN_BYTES", str(thr))
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as hm:
        want = [(t.name, t.dtype, t.shape, t.nbytes, t.file, t.offset) for t in hm.tensors]
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_MAP_LARGE) as h:
        assert [(t.name, t.dtype, t.shape, t.nbytes, t.file, t.offset) for t in h.tensors] == want
        for t in h.tensors:
            assert (t.host_ptr != 0) == (sizes[t.file] >= thr), (t.name, sizes[t.file])
        maps = [l for l in open("/proc/self/maps") if str(tmp_path) in l]
        assert len({l.split()[-1] for l in maps}) == sum(s >= thr for s in sizes)
        # the mappings hold the files' bytes
        import ctypes
        for t in h.tensors:
            if t.host_ptr and t.nbytes:
                with open(ck.paths[t.file], "rb") as fh:
                    fh.seek(t.offset)
                    assert ctypes.string_at(t.host_ptr, min(4096, t.nbytes)) == fh.read(min(4096, t.nbytes))
        t = h.open_times()
        assert t["files_mapped"] == sum(s >= thr for s in sizes) and t["files_registered"] == 0
        assert t["index_ms"] > 0 and t["index_cpu_ms"] > 0 and t["map_cpu_ms"] > 0
        assert t["prefault_ms"] == 0 and t["route_ms"] == 0  # host-only: no route probe
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_NOMAP) as h:
        t = h.open_times()
        assert t["files_mapped"] == 0 and t["map_cpu_ms"] == 0 and t["index_cpu_ms"] > 0
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_PREFAULT) as h:
        t = h.open_times()
        assert t["files_mapped"] == len(sizes) and t["prefault_ms"] > 0
    for bad in (wt.WT_OPEN_NOMAP,):
        with pytest.raises(wt.WtError) as ei:
            wt.Handle(ck.paths, wt.WT_OPEN_MAP_LARGE | bad)
        assert ei.value.code == wt.WT_EINVAL
    monkeypatch.setenv("WT_MAP_MIN_BYTES", "1M")
    with pytest.raises(wt.WtError) as ei:
        wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_MAP_LARGE)
    assert ei.value.code == wt.WT_EINVAL and "WT_MAP_MIN_BYTES" in str(ei.value)


def test_stamps_query_on_host_only_handle(L, tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    # STAMPS is a known flag; a host-only handle launches nothing, so it records no stamps
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_STAMPS) as h:
        with pytest.raises(wt.WtError) as ei:
            h.pass_stamps()
        assert ei.value.code == wt.WT_EINVAL
    with pytest.raises(wt.WtError) as ei:
        wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | (1 << 12))  # unknown flag bit
    assert ei.value.code == wt.WT_EINVAL


def test_nomap_open_parses_without_mapping(L, tmp_path):
    ck = synth.build("many", str(tmp_path / "nm"), n_matrices=5)
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as hm:
        want = [(t.name, t.dtype, t.shape, t.nbytes, t.file, t.offset) for t in hm.tensors]
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY | wt.WT_OPEN_NOMAP) as h:
        assert [(t.name, t.dtype, t.shape, t.nbytes, t.file, t.offset) for t in h.tensors] == want
        assert all(t.host_ptr == 0 for t in h.tensors)
        assert not [l for l in open("/proc/self/maps") if str(tmp_path) in l]  # nothing mapped
        with pytest.raises(wt.WtError) as ei:
            h.residency()
        assert ei.value.code == wt.WT_ENOTSUP
    for bad in (wt.WT_ROUTE_REGISTER, wt.WT_ROUTE_DIRECT, wt.WT_OPEN_PREFAULT):
        with pytest.raises(wt.WtError) as ei:
            wt.Handle(ck.paths, wt.WT_OPEN_NOMAP | bad)
        assert ei.value.code == wt.WT_EINVAL
