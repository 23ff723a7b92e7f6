"""Host-side fault injection (WT_FAULT="<site>[:<n>]"): the n-th open / pread / mmap of a
call fails as if the system call had.  Every failure must return an error status and leave
nothing open or mapped; the library works again once the variable is cleared.  No GPU is
involved (host-only handles and host capsules)."""
import os

import numpy as np
import pytest

from paper_2608_12114_gb300 import build, synth, wt

PAGE = os.sysconf("SC_PAGE_SIZE")


@pytest.fixture(scope="module")
def L():
    build.build()
    return wt.lib()


@pytest.fixture
def fault(monkeypatch):
    def set_(v):
        monkeypatch.setenv("WT_FAULT", v)
    yield set_
    monkeypatch.delenv("WT_FAULT", raising=False)


def mapped(path):
    return [l for l in open("/proc/self/maps") if path in l]


@pytest.mark.parametrize("site,code", [("open", wt.WT_EIO), ("pread", wt.WT_EIO), ("mmap", wt.WT_EIO)])
def test_injected_open_failures_leak_nothing(L, tmp_path, fault, site, code):
    ck = synth.build("many", str(tmp_path / "m"), n_matrices=12)
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()   # warm the pool before counting fds
    fds = len(os.listdir("/proc/self/fd"))
    for n in (1, 7, len(ck.paths)):
        fault("%s:%d" % (site, n))
        with pytest.raises(wt.WtError) as ei:
            wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)
        assert ei.value.code == code and "injected fault" in str(ei.value)
        assert len(os.listdir("/proc/self/fd")) == fds
        assert not mapped(str(tmp_path))
    fault("")
    with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:      # cleared: works again
        assert h.n_files == len(ck.paths)


def test_fault_counter_restarts_when_the_variable_changes(L, tmp_path, fault):
    ck = synth.build("tiny", str(tmp_path))
    fault("open:2")
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()       # first open passes
    with pytest.raises(wt.WtError):
        wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)          # second fails
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()       # third passes again
    fault("open:1")                                          # new value: counting restarts
    with pytest.raises(wt.WtError):
        wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY)
    fault("pread:5")                                          # another site: opens pass
    wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY).close()


def test_injected_mmap_in_the_producer(L, tmp_path, fault):
    p = str(tmp_path / "t.bin")
    np.zeros(PAGE, np.uint8).tofile(p)
    fault("mmap")
    with pytest.raises(wt.WtError) as ei:
        wt.FileTensor.from_file(p, wt.WT_U8, 1, PAGE, wt.WT_DLPACK_HOST)
    assert ei.value.code == wt.WT_EIO
    assert wt.dlpack_live() == 0 and not mapped(p)
