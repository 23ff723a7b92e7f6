"""The map endpoint (Sec. 8.1, contract C1): the GEMV reads W in place from the file mapping
over the host link.  Parity against the oracle, determinism, mixing with resident matrices
in one pass, refusals, and Algorithm 2 measured on this GPU."""
import pytest

import oracle
from paper_2608_12114_gb300 import build, pipeline, policy, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def mapped_descs(torch, h, xs, ys, only=None):
    out = []
    for i, t in enumerate(h.tensors):
        if len(t.shape) != 2 or (only is not None and i not in only):
            continue
        M, K = t.shape
        out.append(wt.gemv_desc(t.host_ptr, t.dtype, M, K, xs[(K, t.dtype)].data_ptr(), ys[i].data_ptr()))
    return out


def inputs(torch, h):
    xs, ys = {}, {}
    for i, t in enumerate(h.tensors):
        if len(t.shape) == 2:
            key = (t.shape[1], t.dtype)
            if key not in xs:
                xs[key] = torch.from_numpy(synth.make_x(t.shape[1], t.dtype)).cuda()
            ys[i] = torch.full((t.shape[0],), float("nan"), dtype=torch.float32, device="cuda")
    torch.cuda.synchronize()
    return xs, ys


SHAPES = [(1, 8), (7, 24), (33, 40), (100, 256), (65, 264), (17, 2048), (9, 2056), (5, 4096),
          (3, 16384), (4, 100000), (2, 7), (6, 0)]


@pytest.mark.parametrize("dtype", [synth.DT_BF16, synth.DT_F16, synth.DT_F32])
def test_mapped_gemv_matches_oracle(torch, tmp_path, dtype):
    ck = synth.write_files(synth.custom(str(tmp_path), SHAPES, dtype=dtype, name="m%d" % dtype))
    co = oracle.CheckpointOracle(ck.paths)
    with wt.Handle(ck.paths, wt.WT_OPEN_PREFAULT) as h:
        xs, ys = inputs(torch, h)
        h.pass_(mapped_descs(torch, h, xs, ys), 0)
        torch.cuda.synchronize()
        y1 = {i: y.clone() for i, y in ys.items()}
        h.pass_(mapped_descs(torch, h, xs, ys), 0)
        torch.cuda.synchronize()
        for i, t in enumerate(h.tensors):
            M, K = t.shape
            yhat, a = oracle.gemv(co.files[0].blob(i), t.dtype, M, K, synth.make_x(K, t.dtype))
            err = oracle.gemv_error(ys[i].cpu().numpy(), yhat, a)
            assert err <= TOL, (t.name, err)
            assert torch.equal(y1[i], ys[i])  # deterministic run to run
        assert h.device_status() == 0


def test_mapped_and_resident_in_one_pass(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path), layers=1, vocab=700)
    co = oracle.CheckpointOracle(ck.paths)
    with wt.Handle(ck.paths) as h:
        mats = pipeline.matrices(h)
        dev = pipeline.DeviceCheckpoint.allocate(h, mats)
        xs, ys_dev = dev.inputs(), dev.outputs()
        torch.cuda.synchronize()
        dev.adopt(h, wt.WT_ADOPT_GATHER, 0)
        torch.cuda.synchronize()
        res = dev.descs(xs, ys_dev)
        ys_map = {k: torch.empty_like(y) for k, y in ys_dev.items()}
        mixed = []
        for n, k in enumerate(dev.gemv_mats()):
            t = h.tensors[mats[k].parts[0]]
            if n % 2:
                mixed.append(wt.gemv_desc(t.host_ptr, t.dtype, t.shape[0], t.shape[1],
                                          xs[(t.shape[1], t.dtype)].data_ptr(), ys_map[k].data_ptr()))
            else:
                r = res[n]
                mixed.append(wt.gemv_desc(int(r["W"]), int(r["dtype"]), int(r["M"]), int(r["K"]), int(r["x"]),
                                          ys_map[k].data_ptr()))
        torch.cuda.synchronize()
        h.pass_(res, 0)
        h.pass_(mixed, 0)
        torch.cuda.synchronize()
        for n, k in enumerate(dev.gemv_mats()):
            m = mats[k]
            t = h.tensors[m.parts[0]]
            W = co.blob_of(t.file, t.name)
            yhat, a = oracle.gemv(W, m.dtype, m.shape[0], m.shape[1], synth.make_x(m.shape[1], m.dtype))
            assert oracle.gemv_error(ys_map[k].cpu().numpy(), yhat, a) <= TOL, m.name
            assert oracle.gemv_error(ys_dev[k].cpu().numpy(), yhat, a) <= TOL, m.name
            if n % 2 == 0:
                assert torch.equal(ys_map[k], ys_dev[k])  # resident rows: same kernel, same bits


def test_refusals(torch, tmp_path):
    ck = synth.write_files(synth.custom(str(tmp_path), [(8, 64), (8, 64)], name="r"))
    with wt.Handle(ck.paths) as h:
        xs, ys = inputs(torch, h)
        t0, t1 = h.tensors
        x = xs[(64, t0.dtype)].data_ptr()
        with pytest.raises(wt.WtError) as ei:  # y inside the read-only mapping
            h.pass_([wt.gemv_desc(t0.host_ptr, t0.dtype, 8, 64, x, t1.host_ptr)], 0)
        assert ei.value.code == wt.WT_EINVAL
        size = t1.offset + t1.nbytes
        start = t1.host_ptr - t1.offset
        with pytest.raises(wt.WtError) as ei:  # W running past the end of the mapping
            h.pass_([wt.gemv_desc(start + size - 64, t0.dtype, 8, 64, x, ys[0].data_ptr())], 0)
        assert ei.value.code == wt.WT_EINVAL
    with wt.Handle(ck.paths, wt.WT_ROUTE_NONE) as h:
        xs, ys = inputs(torch, h)
        t0 = h.tensors[0]
        with pytest.raises(wt.WtError) as ei:  # no device route to the mapping
            h.pass_([wt.gemv_desc(t0.host_ptr, t0.dtype, 8, 64, xs[(64, t0.dtype)].data_ptr(),
                                  ys[0].data_ptr())], 0)
        assert ei.value.code == wt.WT_ENOTSUP


def test_algorithm2_on_this_gpu(torch, tmp_path):
    ck = synth.build("mid", str(tmp_path), layers=2, workers=4)
    out = policy.measure_gb300(ck.paths, reps=3)
    assert out.resident_before == out.resident_after
    assert set(out.rates_gbs) == set(policy.ENDPOINTS)
    # the host link caps map and copy; HBM makes the resident arm far faster
    assert out.rates_gbs["resident"] > 5 * max(out.rates_gbs["map"], out.rates_gbs["copy"])
    assert out.decision == "resident"
