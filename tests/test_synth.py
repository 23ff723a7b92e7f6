"""The seeded workloads have the shapes, sizes and structure they are meant to have."""

import numpy as np

from paper_2608_12114_gb300 import synth


def test_decoder_byte_totals():
    mid = synth.decoder("/nonexistent", "mid")
    large = synth.decoder("/nonexistent", "large")
    assert mid.data_bytes == 5_403_120_640 and len(mid.paths) == 3
    assert large.data_bytes == 16_060_522_496 and len(large.paths) == 4
    assert mid.weight_bytes == 5_402_787_840 and large.weight_bytes == 16_059_990_016
    assert len(mid.tensors) == len(large.tensors) == 291
    assert len(mid.matrices) == len(large.matrices) == 226
    k = [m for m in large.matrices if m.name == "layers.0.k"][0]
    assert (k.M, k.K) == (1024, 4096)
    down = [m for m in large.matrices if m.name == "layers.3.down"][0]
    assert (down.M, down.K) == (4096, 14336)
    assert large.matrices[0].name == "embed" and large.matrices[-1].name == "lm_head"
    # greedy shards: every shard but the last stays within ceil(total / n)
    for ck in (mid, large):
        cap = -(-ck.data_bytes // len(ck.paths))
        for f in range(len(ck.paths) - 1):
            ts = [ck.tensors[i] for i in ck.file_tensors(f)]
            assert sum(t.nbytes for t in ts) <= cap


def test_many_structure():
    ck = synth.many("/nonexistent")
    assert len(ck.matrices) == 1253 and len(ck.paths) == 2506 and len(ck.tensors) == 2506
    for m in ck.matrices:
        assert m.K in (32, 64, 128, 256, 512, 1024, 2048)
        assert m.M % 2 == 0
        half = m.M // 2 * m.K * 2
        assert half <= 4 * 1024 * 1024 and (half >= 4096 // 2 or m.M == 2)
    assert 1.2e9 < ck.data_bytes < 1.9e9


def test_sweep_sizes():
    ck = synth.sweep("/nonexistent")
    sizes = [t.nbytes for t in ck.tensors]
    assert sizes == [1 << (20 + i) for i in range(14)]


def test_x_and_files_are_deterministic(tmp_path):
    assert np.array_equal(synth.make_x(4096, synth.DT_BF16), synth.make_x(4096, synth.DT_BF16))
    assert not np.array_equal(synth.make_x(4096, synth.DT_BF16)[:64], synth.make_x(2048, synth.DT_BF16)[:64])
    a = synth.build("mid", str(tmp_path / "a"), layers=1, vocab=40)
    b = synth.build("mid", str(tmp_path / "b"), layers=1, vocab=40, )
    for pa, pb in zip(a.paths, b.paths):
        assert open(pa, "rb").read() == open(pb, "rb").read()


def test_parallel_writer_matches_serial(tmp_path):
    a = synth.build("many", str(tmp_path / "s"), n_matrices=6)
    b = synth.build("many", str(tmp_path / "p"), n_matrices=6, workers=3)
    for pa, pb in zip(a.paths, b.paths):
        assert open(pa, "rb").read() == open(pb, "rb").read()


def test_bf16_rounding_is_nearest_even():
    f = np.array([1.0, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -8, -1.5, 2 ** -133], np.float32)
    bits = synth.f32_to_bf16_bits(f)
    # 1+2^-8 is a tie between 0x3F80 and 0x3F81 -> even (0x3F80); 1+3*2^-8 -> 0x3F82
    assert list(bits) == [0x3F80, 0x3F80, 0x3F82, 0xBFC0, 0x0001]
