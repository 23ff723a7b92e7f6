"""Parity at the workloads' full sizes, in the launch configuration bench.py times.

For each workload: file -> first use exactly as the bench's e2e leg runs it (gather
ingest on one stream, event-gated grouped GEMV launches on another), then the resident
pass exactly as the bench's timed step runs it (every matrix in one launch).  Checked:
  - the two passes give bitwise-identical y (row results do not depend on grouping);
  - D_tree of every ingested tensor equals the oracle's, and D_plain where the GPU computes it
    (up to 256 MiB); above that, a seeded 1 % of the 4 KiB leaves is compared byte for byte;
  - sampled GEMV rows (first, last and 16 seeded rows of every matrix) against the fp64
    oracle, max |y - yhat| / sum|W x| <= 2e-3; the many-small workload is checked on every row.
"""
import shutil

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, pipeline, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def run_and_check(torch, ck, rows=16, plain_limit=256 << 20):
    co = oracle.CheckpointOracle(ck.paths)
    h = wt.Handle(ck.paths)
    try:
        dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
        xs, ys = dev.inputs(), dev.outputs()
        ingest_s, consume_s = torch.cuda.Stream(), torch.cuda.Stream()
        torch.cuda.synchronize()
        ev = dev.adopt(h, wt.WT_ADOPT_GATHER, ingest_s.cuda_stream)
        h.pass_(dev.descs(xs, ys, ev), consume_s.cuda_stream)          # first use
        consume_s.synchronize()
        ingest_s.synchronize()
        first = {k: y.clone() for k, y in ys.items()}
        torch.cuda.synchronize()
        h.pass_(dev.descs(xs, ys), consume_s.cuda_stream)              # resident pass
        consume_s.synchronize()
        for k in ys:
            assert torch.equal(first[k], ys[k]), dev.mats[k].name
        assert h.device_status() == 0

        # bytes: D_tree of every tensor (and D_plain up to plain_limit)
        idx = list(range(len(h.tensors)))
        out = torch.zeros(len(idx), dtype=torch.int64, device="cuda")
        h.checksum([dev.dst[i] for i in idx], [h.tensors[i].nbytes for i in idx], out.data_ptr(), 0)
        tree = [int(v) & (2 ** 64 - 1) for v in out.cpu().tolist()]
        small = [i for i in idx if h.tensors[i].nbytes <= plain_limit]
        outp = torch.zeros(max(1, len(small)), dtype=torch.int64, device="cuda")
        h.checksum([dev.dst[i] for i in small], [h.tensors[i].nbytes for i in small], outp.data_ptr(), 0,
                   plain=True)
        plain = dict(zip(small, [int(v) & (2 ** 64 - 1) for v in outp.cpu().tolist()]))
        where = {}  # tensor -> (device buffer, byte offset in it)
        for k, m in enumerate(dev.mats):
            for i in m.parts:
                where[i] = (dev.bufs[k], dev.dst[i] - dev.bufs[k].data_ptr())
        rng = np.random.default_rng(99)
        for i, t in enumerate(h.tensors):
            fo = co.files[t.file]
            blob = fo.blob([e["name"] for e in fo.entries].index(t.name))
            assert tree[i] == oracle.fnv_tree(blob), t.name
            if i in plain:
                assert plain[i] == oracle.fnv1a64(blob), t.name
            elif i in where:
                # beyond the literal digest's size: the leaf tree plus a byte compare of a seeded
                # 1 % of the 4 KiB leaves (at least 16), read back from the device
                nleaf = (t.nbytes + 4095) // 4096
                buf, off = where[i]
                for lf in rng.choice(nleaf, max(16, nleaf // 100), replace=False):
                    a, b = int(lf) * 4096, min(int(lf) * 4096 + 4096, t.nbytes)
                    assert np.array_equal(buf[off + a:off + b].cpu().numpy(), blob[a:b]), (t.name, int(lf))

        # GEMV: sampled rows (or all rows when rows is None)
        worst = 0.0
        for k in dev.gemv_mats():
            m = dev.mats[k]
            M, K = m.shape
            W = co.matrix_bytes([(h.tensors[i].file, h.tensors[i].name) for i in m.parts])
            x = synth.make_x(K, m.dtype)
            y = ys[k].cpu().numpy().astype(np.float64)
            if rows is None:
                yhat, a = oracle.gemv(W, m.dtype, M, K, x)
                err = oracle.gemv_error(y, yhat, a)
            else:
                r = sorted({0, M - 1} | {int(v) for v in np.random.default_rng(k).integers(0, M, rows)})
                yhat, a = oracle.gemv_rows(W, m.dtype, M, K, x, r)
                err = oracle.gemv_error(y[r], yhat, a)
            assert err <= TOL, (m.name, err)
            worst = max(worst, err)
        return worst
    finally:
        h.close()
        co.close()


def test_large_decoder_full_size(torch, tmp_path):
    ck = synth.build("large", str(tmp_path), workers=16)
    assert ck.data_bytes == 16_060_522_496
    try:
        worst = run_and_check(torch, ck)
        assert worst < 1e-4  # fp32 accumulation of K <= 14336 products stays far inside 2e-3
    finally:
        shutil.rmtree(str(tmp_path), ignore_errors=True)


def test_mid_decoder_full_size(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path), workers=16)
    assert ck.data_bytes == 5_403_120_640
    try:
        run_and_check(torch, ck)
    finally:
        shutil.rmtree(str(tmp_path), ignore_errors=True)


def test_many_small_full_size_every_row(torch, tmp_path):
    ck = synth.build("many", str(tmp_path), workers=16)
    assert len(ck.paths) == 2506
    try:
        run_and_check(torch, ck, rows=None)
    finally:
        shutil.rmtree(str(tmp_path), ignore_errors=True)


def test_sweep_points_full_size(torch, tmp_path):
    """1 MiB, 64 MiB, 1 GiB and 8 GiB (K = 1,048,576: split-K tiles, rows of 2 MiB)."""
    ck = synth.build("sweep", str(tmp_path), points=[0, 6, 10, 13], workers=16)
    try:
        run_and_check(torch, ck)
    finally:
        shutil.rmtree(str(tmp_path), ignore_errors=True)


def test_matched_protocol_int8_full_size(torch, tmp_path):
    """The paper's matched protocol: 12 files of 12288x7168 int8 (88.1 MB) with fp16 row scales."""
    ck = synth.build("protocol_q8", str(tmp_path), workers=16)
    co = oracle.CheckpointOracle(ck.paths)
    h = wt.Handle(ck.paths)
    try:
        dev = pipeline.DeviceCheckpoint.allocate(h, pipeline.matrices(h))
        xs, ys = dev.inputs(), dev.outputs()
        ingest_s, consume_s = torch.cuda.Stream(), torch.cuda.Stream()
        torch.cuda.synchronize()
        ev = dev.adopt(h, wt.WT_ADOPT_GATHER, ingest_s.cuda_stream)
        h.pass_(dev.descs(xs, ys, ev), consume_s.cuda_stream)
        consume_s.synchronize()
        ingest_s.synchronize()
        first = {k: y.clone() for k, y in ys.items()}
        h.pass_(dev.descs(xs, ys), consume_s.cuda_stream)
        consume_s.synchronize()
        assert len(ys) == 12 and all(torch.equal(first[k], ys[k]) for k in ys)
        for k in dev.gemv_mats():
            m = dev.mats[k]
            t, sc = h.tensors[m.parts[0]], h.tensors[m.scale]
            r = sorted({0, 12287} | {int(v) for v in np.random.default_rng(k).integers(0, 12288, 16)})
            yhat, a = oracle.gemv_q8(co.blob_of(t.file, t.name), co.blob_of(sc.file, sc.name), 12288, 7168,
                                     synth.make_x(7168, synth.DT_I8), rows=r)
            assert oracle.gemv_error(ys[k].cpu().numpy()[r], yhat, a) <= TOL
        assert h.device_status() == 0
    finally:
        h.close()
        co.close()
        shutil.rmtree(str(tmp_path), ignore_errors=True)
