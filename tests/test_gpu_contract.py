"""The contract ablation (Sec. 4, Table "cube"): every one of the eight C1/C2/C3 cells and
every ordering mechanism computes the same GEMV outputs, each within tolerance of the oracle;
cells that read W the same way give identical bits."""
import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import build, contract, synth, wt

pytestmark = pytest.mark.gpu
TOL = 2e-3


@pytest.fixture(scope="module")
def torch():
    import torch
    assert torch.cuda.is_available()
    build.build()
    wt.lib()
    return torch


def test_every_cell_and_ordering_gives_the_oracle_result(torch, tmp_path):
    ck = synth.build("protocol", str(tmp_path), matrices=4, rows=300, cols=520)
    co = oracle.CheckpointOracle(ck.paths)
    want = []
    for f in range(4):
        yhat, a = oracle.gemv(co.blob_of(f, "w"), synth.DT_BF16, 300, 520, synth.make_x(520, synth.DT_BF16))
        want.append((yhat, a))
    c = contract.Contract(ck.paths)
    try:
        got = {}
        for cell in contract.CELLS:
            for y in c.y_dev:
                y.fill_(float("nan"))
            torch.cuda.synchronize()
            c.run_pass(*cell)
            torch.cuda.synchronize()
            got[cell] = [np.array(v, copy=True) for v in c.outputs(cell[1])]
            for (yhat, a), y in zip(want, got[cell]):
                assert oracle.gemv_error(y, yhat, a) <= TOL, contract.cell_name(cell)
        for cell in contract.CELLS:  # same W route -> same kernel -> same bits
            ref = got[(cell[0], 1, 1)]
            assert all(np.array_equal(a, b) for a, b in zip(got[cell], ref)), contract.cell_name(cell)
        fw = torch.cuda.current_stream()
        for mech in contract.ORDERINGS:
            for y in c.y_dev:
                y.fill_(float("nan"))
            torch.cuda.synchronize()
            c.run_ordered(mech, fw)
            torch.cuda.synchronize()
            out = c.outputs(1)
            assert all(np.array_equal(a, b) for a, b in zip(out, got[(1, 1, 1)])), mech
    finally:
        c.close()
