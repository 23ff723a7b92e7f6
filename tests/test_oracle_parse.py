"""Pins for the oracle's parser (O1): hand-built files, every rejection rule, round trips."""
import os

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import synth
from tests import _files


def write(tmp, name, data):
    p = os.path.join(tmp, name)
    with open(p, "wb") as f:
        f.write(data)
    return p


def test_hand_built_two_entries(tmp_path):
    img, (o1, ba), (o2, bb) = _files.good_two_entry()
    f = oracle.load(write(str(tmp_path), "g.wt", img))
    assert [e["name"] for e in f.entries] == ["a", "b"]
    assert f.entries[0]["shape"] == (2, 4) and f.entries[1]["shape"] == (3,)
    assert f.entries[0]["dtype"] == 1 and f.entries[0]["offset"] == o1 and f.entries[1]["offset"] == o2
    assert f.blob(0).tobytes() == ba and f.blob(1).tobytes() == bb


@pytest.mark.parametrize("label,img", _files.bad_files(), ids=[b[0] for b in _files.bad_files()])
def test_rejections(tmp_path, label, img):
    with pytest.raises(oracle.OracleError):
        oracle.load(write(str(tmp_path), label + ".wt", img))


def test_missing_file(tmp_path):
    with pytest.raises(oracle.OracleError):
        oracle.load(os.path.join(str(tmp_path), "nope.wt"))


def test_zero_size_tensor_and_empty_index(tmp_path):
    e = _files.entry("z", 1, (0, 8), 64, 0)
    f = oracle.load(write(str(tmp_path), "z.wt", _files.assemble([e], [], pad_to=64)))
    assert f.entries[0]["nbytes"] == 0 and f.entries[0]["shape"] == (0, 8)
    f = oracle.load(write(str(tmp_path), "e.wt", _files.assemble([], [])))
    assert f.entries == []


def test_round_trip_tiny(tmp_path):
    ck = synth.build("tiny", str(tmp_path))
    f = oracle.load(ck.paths[0])
    assert len(f.entries) == len(ck.tensors) == 16
    for i, (e, t) in enumerate(zip(f.entries, ck.tensors)):
        assert (e["name"], e["dtype"], e["shape"], e["offset"], e["nbytes"]) == \
               (t.name, t.dtype, t.shape, t.offset, t.nbytes)
        assert e["offset"] % 64 == 0
        assert f.blob(i).tobytes() == t.array.astype("<f4").tobytes()
    assert ck.data_bytes == 2105344


def test_round_trip_decoder_shards(tmp_path):
    ck = synth.build("mid", str(tmp_path), layers=1, vocab=64)
    seen = 0
    for fi, p in enumerate(ck.paths):
        f = oracle.load(p)
        ts = [t for t in ck.tensors if t.file == fi]
        assert [e["name"] for e in f.entries] == [t.name for t in ts]
        for e, t in zip(f.entries, ts):
            assert e["shape"] == t.shape and e["nbytes"] == t.nbytes and e["offset"] == t.offset
            if t.fill == "ones":
                assert np.all(f.blob(f.entries.index(e)).view("<u2") == 0x3F80)
        seen += len(ts)
    assert seen == len(ck.tensors) == 1 + 9 + 2


def test_many_halves_are_row_blocks(tmp_path):
    ck = synth.build("many", str(tmp_path), n_matrices=5)
    co = oracle.CheckpointOracle(ck.paths)
    for m in ck.matrices:
        W = co.matrix_bytes([(ck.tensors[i].file, ck.tensors[i].name) for i in m.parts])
        assert W.size == m.M * m.K * 2
        assert ck.tensors[m.parts[0]].shape == (m.M // 2, m.K)
        assert ck.tensors[m.parts[1]].shape == (m.M - m.M // 2, m.K)
