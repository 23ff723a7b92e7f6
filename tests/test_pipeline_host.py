"""Host-side bookkeeping of the first use (no GPU): the io region's layout, by which one
allocation and one host-to-device copy serve every x and one device-to-host copy every y."""
import numpy as np
import pytest

from paper_2608_12114_gb300 import build, pipeline, synth, wt


def test_io_layout(tmp_path):
    build.build()
    for workload, kw in (("many", {"n_matrices": 30}), ("protocol_q8", {"matrices": 2, "rows": 256, "cols": 512}),
                         ("tiny", {})):
        ck = synth.build(workload, str(tmp_path / workload), **kw)
        with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
            mats = pipeline.matrices(h)
        xs, y_off, rows, total = pipeline.io_layout(mats)
        g = [m for m in mats if m.gemv]
        assert rows == [m.shape[0] for m in g] and total == y_off + 4 * sum(rows)
        assert set(xs) == {(m.shape[1], m.dtype) for m in g}
        spans = sorted(xs.values())
        for (o, n), (K, dt) in zip(spans, sorted(xs, key=xs.get)):
            assert o % 256 == 0 and n == K * (2 if dt == wt.WT_I8 else {wt.WT_F32: 4}.get(dt, 2))
        for (o, n), (o2, _) in zip(spans, spans[1:]):
            assert o + n <= o2                      # no two x overlap
        assert y_off % 256 == 0 and y_off >= spans[-1][0] + spans[-1][1]


def write_entries(path, specs):
    """A checkpoint file of (name, dtype, shape) entries with zero bytes (tests._files encoder)."""
    from tests import _files
    es = {0: 4, 1: 2, 2: 2, 3: 1, 4: 1}
    sizes = [int(np.prod(sh)) * es[dt] for _, dt, sh in specs]
    hl = _files.header_len([_files.entry(n, dt, sh, 0, nb) for (n, dt, sh), nb in zip(specs, sizes)])
    pos, ents, blobs = _files.aligned(hl), [], []
    for (n, dt, sh), nb in zip(specs, sizes):
        ents.append(_files.entry(n, dt, sh, pos, nb))
        blobs.append((pos, bytes(nb)))
        pos = _files.aligned(pos + nb)
    with open(path, "wb") as f:
        f.write(_files.assemble(ents, blobs))


def test_matrices_columns_match_the_reference_grouping(tmp_path):
    build.build()
    # both branches of the grouping: plain loops up to 32 tensors, numpy columns above
    cases = [("many", {"n_matrices": 60}), ("many", {"n_matrices": 10}),
             ("protocol_q8", {"matrices": 3, "rows": 64, "cols": 256}),
             ("protocol_q8", {"matrices": 20, "rows": 64, "cols": 256}),
             ("tiny", {}), ("mid", {"layers": 1}), ("mid", {"layers": 4})]
    for workload, kw in cases:
        ck = synth.build(workload, str(tmp_path / workload), **kw)
        with wt.Handle(ck.paths, wt.WT_OPEN_HOST_ONLY) as h:
            m, ref = pipeline.matrices(h), pipeline._matrices_list(h)
        assert len(m) == len(ref)
        for k, r in enumerate(ref):
            got = m[k]
            assert (got.name, got.dtype, tuple(got.shape), got.parts, got.gemv, got.scale) == \
                   (r.name, r.dtype, tuple(r.shape), r.parts, r.gemv, r.scale), (workload, k)
        assert m.nbytes.tolist() == [sum(h.tensors.nbytes[i] for i in r.parts) for r in ref]
    # hand-built: blocks out of order and across files, plain tensors named like blocks ("v#rx",
    # and a ten-digit block number), a nine-digit block number, an int8 matrix with row scales
    p1, p2 = str(tmp_path / "a.wt"), str(tmp_path / "b.wt")
    write_entries(p1, [("w#r1", 1, (3, 8)), ("v#rx", 1, (4,)), ("n", 2, (5,)), ("u#r123456789", 1, (2, 8)),
                    ("t#r1234567890", 1, (2, 8))])
    write_entries(p2, [("w#r0", 1, (2, 8)), ("q", 3, (4, 16)), ("q.scale", 2, (4,)), ("w#r2", 1, (1, 8))])
    with wt.Handle([p1, p2], wt.WT_OPEN_HOST_ONLY) as h:
        m, ref = pipeline.matrices(h), pipeline._matrices_list(h)
        got = [(r.name, tuple(r.shape), r.parts, r.gemv, r.scale) for r in m]
        assert got == [(r.name, tuple(r.shape), r.parts, r.gemv, r.scale) for r in ref]
        assert got[0] == ("w", (6, 8), [5, 0, 8], True, None) and ("q", (4, 16), [6], True, 7) in got
        assert ("t#r1234567890", (2, 8), [4], True, None) in got
    # row blocks that do not stack are refused, as by the reference grouping
    lone = [("a#r0", 1, (16,))] + [("p%d" % i, 1, (4,)) for i in range(40)]  # no two joined, numpy branch
    for bad in ([("a#r0", 1, (2, 8)), ("a#r1", 1, (2, 9))], [("a#r0", 1, (2, 8)), ("a#r1", 2, (2, 8))],
                [("a#r0", 1, (2, 8)), ("a#r1", 1, (16,))], [("a#r0", 1, (16,))], lone,
                lone + [("a#r1", 1, (2, 8))]):
        p = str(tmp_path / "bad.wt")
        write_entries(p, bad)
        with wt.Handle([p], wt.WT_OPEN_HOST_ONLY) as h:
            with pytest.raises(ValueError):
                pipeline.matrices(h)
            with pytest.raises(ValueError):
                pipeline._matrices_list(h)


def test_segment_bounds_match_the_running_sum():
    def reference(sizes, first, growth):
        total = sum(sizes)
        seg = total if total < (2 << 30) else min(first, total)
        cuts, acc, limit = [], 0, seg
        for k, n in enumerate(sizes):
            acc += n
            if acc >= limit and k + 1 < len(sizes):
                cuts.append(k + 1)
                seg = int(seg * growth)
                limit = acc + seg
        return [0] + cuts + [len(sizes)]
    rng = np.random.default_rng(4)
    for t in range(300):
        n = int(rng.integers(0, 400))
        sizes = rng.choice([0, 64, 1 << 20, 50 << 20, 300 << 20, 1 << 30], n) * rng.integers(0, 3, n)
        first, growth = int(rng.choice([1 << 20, 256 << 20])), float(rng.choice([1.5, 2.0]))
        assert pipeline.segment_bounds(np.asarray(sizes, np.int64), first, growth) == \
               reference(sizes.tolist(), first, growth), t


class _Buf:
    def __init__(self, p):
        self.p = p

    def data_ptr(self):
        return self.p


def test_descs_and_addresses_follow_the_adoption_order(tmp_path):
    """Each descriptor waits on the event of the matrix's last-adopted tensor (a row block or
    its row scales), and row blocks sit back to back in their matrix's buffer."""
    build.build()
    ck = synth.build("many", str(tmp_path / "m"), n_matrices=50)
    ckq = synth.build("protocol_q8", str(tmp_path / "q"), matrices=3, rows=64, cols=256)
    rng = np.random.default_rng(9)
    cks = synth.build("many", str(tmp_path / "s"), n_matrices=8)
    ckq2 = synth.build("protocol_q8", str(tmp_path / "q2"), matrices=20, rows=64, cols=256)
    for paths in (ck.paths, ckq.paths, cks.paths, ckq2.paths):  # large and small branches
        with wt.Handle(paths, wt.WT_OPEN_HOST_ONLY) as h:
            mats = pipeline.matrices(h)
            dc = pipeline.DeviceCheckpoint._new(h, mats, None)
            dc.ptrs[:] = (1 << 40) + np.arange(len(mats), dtype=np.uint64) * (1 << 24)
            dc._set_dst(h)
            for k, m in enumerate(mats):
                off = 0
                for i in m.parts:
                    assert dc.dst[i] == int(dc.ptrs[k]) + off
                    off += h.tensors.nbytes[i]
            order = rng.permutation(len(h.tensors))
            ev = pipeline.ReadyEvents(len(h.tensors))
            ev.add(order[:len(order) // 2], 1000 + order[:len(order) // 2])
            ev.add(order[len(order) // 2:], 1000 + order[len(order) // 2:])
            ks = dc.gemv_mats()
            xs = {key: 7000 + 64 * j for j, key in enumerate(pipeline.io_layout(mats)[0])}
            ys = pipeline.FlatOutputs(_Buf(1 << 36), ks, [int(mats.M[k]) for k in ks])
            d = dc.descs(xs, ys, ev)
            rank = {int(t): n for n, t in enumerate(order)}
            for j, k in enumerate(ks):
                m = mats[k]
                ts = m.parts + ([m.scale] if m.scale is not None else [])
                last = max(ts, key=rank.__getitem__)
                assert int(d["wait_event"][j]) == 1000 + last
                assert int(d["W"][j]) == int(dc.ptrs[k]) and int(d["x"][j]) == xs[(m.shape[1], m.dtype)]
                assert (int(d["M"][j]), int(d["K"][j])) == m.shape
                assert int(d["scale"][j]) == (dc.dst[m.scale] if m.scale is not None else 0)
            assert d["y"].tolist() == [(1 << 36) + 4 * o for o in ys.offs.tolist()]
            # the same events as a plain mapping give the same waits
            d2 = dc.descs(xs, ys, dict(ev.items()))
            assert np.array_equal(d["wait_event"], d2["wait_event"])


def test_random_checkpoints_group_like_the_reference(tmp_path):
    """Random multi-file checkpoints (row blocks spread over files in any order, plain 1-D and
    2-D tensors, int8 matrices with and without row scales, names that only look like
    blocks): the columnar grouping, the io layout and the buffer offsets equal the plain-Python
    reference's, on both branches (up to 32 tensors and above)."""
    build.build()
    rng = np.random.default_rng(21)
    for trial in range(24):
        specs = []  # (name, dtype, shape)
        for m in range(int(rng.integers(1, 30))):
            kind = rng.integers(0, 5)
            K = int(rng.choice([8, 16, 64, 256]))
            dt = int(rng.choice([0, 1, 2]))
            if kind == 0:    # a matrix split into row blocks
                nb = int(rng.integers(1, 4))
                for b in rng.permutation(nb).tolist():
                    specs.append(("m%d#r%d" % (m, b), dt, (int(rng.integers(1, 5)), K)))
            elif kind == 1:  # a plain 2-D matrix
                specs.append(("p%d" % m, dt, (int(rng.integers(1, 6)), K)))
            elif kind == 2:  # a vector, or a name that only looks like a block
                specs.append(("v%d#r%s" % (m, rng.choice(["x", "", "1234567890"])), dt, (K,)))
            elif kind == 3:  # int8 with fp16 row scales
                M = int(rng.integers(1, 6))
                specs.append(("q%d" % m, 3, (M, K)))
                specs.append(("q%d.scale" % m, 2, (M,)))
            else:            # int8 without scales, and scales of the wrong length
                specs.append(("r%d" % m, 3, (3, K)))
                specs.append(("r%d.scale" % m, 2, (2,)))
        order = rng.permutation(len(specs)).tolist()
        nf = int(rng.integers(1, 4))
        files = [[] for _ in range(nf)]
        for j, i in enumerate(order):
            files[j % nf].append(specs[i])
        paths = []
        for f, fs in enumerate(files):
            if fs:
                p = str(tmp_path / ("t%d_%d.wt" % (trial, f)))
                write_entries(p, fs)
                paths.append(p)
        with wt.Handle(paths, wt.WT_OPEN_HOST_ONLY) as h:
            m, ref = pipeline.matrices(h), pipeline._matrices_list(h)
            got = [(r.name, r.dtype, tuple(r.shape), r.parts, r.gemv, r.scale) for r in m]
            assert got == [(r.name, r.dtype, tuple(r.shape), r.parts, r.gemv, r.scale) for r in ref], trial
            assert pipeline.io_layout(m) == pipeline.io_layout(ref), trial
            dc = pipeline.DeviceCheckpoint._new(h, m, None)
            dc.ptrs[:] = (1 << 40) + np.arange(len(m), dtype=np.uint64) * (1 << 20)
            dc._set_dst(h)
            for k, r in enumerate(ref):
                off = 0
                for i in r.parts:
                    assert dc.dst[i] == (1 << 40) + k * (1 << 20) + off
                    off += h.tensors.nbytes[i]
