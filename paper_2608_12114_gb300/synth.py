"""Seeded synthetic checkpoints and GEMV inputs.

This module only *produces inputs*: it lays out files in the container format
(a length-prefixed index of name/dtype/shape/offset/nbytes, then 64-byte
aligned raw blobs) and fills them with seeded values.  It holds none of the
path's arithmetic (no parsing, no checksum, no GEMV); the CUDA library and the
CPU oracle each decode these files with their own code.

The container stands in for the paper's per-tensor page-aligned files
(Sec. 5.3 suggests an aligned container as the alternative to one inode per
tensor; Algorithm 1 guards size = M*K*sizeof(dtype)).

Layout (all integers little-endian):

    u8  magic[8] = "WTCKPT01"
    u64 index_bytes
    index: u32 n_entries, then per entry
        u16 name_len, u8 name[name_len], u8 dtype, u8 ndim,
        u64 shape[ndim], u64 offset, u64 nbytes
    zero padding; blobs in index order, each at a 64-byte aligned offset

Workloads (shapes of the paper's measured cases; values are synthetic):
  tiny   8 fp32 256x256 matrices + 8 fp32[256] vectors, U[-1,1] from PCG64(0)
  sweep  one bf16 4096 x (128*2^i) matrix per file, N(0, 0.02)
  many   1253 bf16 matrices split by rows into 2506 single-tensor files
         (the 1253-matrix / 2506-file spine shape of Sec. 5.3)
  mid    32-layer decoder, d=2560, FFN 6912, vocab 32000, 3 shards
  large  32-layer decoder, d=4096, kv 1024, FFN 14336, vocab 128256, 4 shards
"""
from __future__ import annotations

import dataclasses
import math
import os
import struct
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

MAGIC = b"WTCKPT01"
ALIGN = 64
DT_F32, DT_BF16, DT_F16, DT_I8, DT_U8 = 0, 1, 2, 3, 4
DTYPE_NAMES = {DT_F32: "f32", DT_BF16: "bf16", DT_F16: "f16", DT_I8: "i8", DT_U8: "u8"}
ELEM_SIZE = {DT_F32: 4, DT_BF16: 2, DT_F16: 2, DT_I8: 1, DT_U8: 1}

# spawn-key prefixes for the per-tensor value streams of each workload
_STREAM_KEY = {"many": 1, "sweep": 2, "mid": 3, "large": 4, "custom": 5, "protocol": 6, "protocol_q8": 7}
_CHUNK = 1 << 24  # elements per value stream (each chunk of a tensor has its own stream)


@dataclasses.dataclass
class TensorSpec:
    """One index entry: where it lives and how its values are drawn."""

    name: str
    dtype: int
    shape: Tuple[int, ...]
    file: int
    fill: str = "normal"          # "normal" (std=scale), "uniform" (+-scale), "ones", "array",
                                  # "int8" (uniform integers in [-127, 127]), "rowscale" (U[scale, 10*scale])
    scale: float = 0.02
    key: Tuple[int, ...] = ()     # spawn key of the value stream
    offset: int = 0               # absolute file offset (filled by layout())
    array: Optional[np.ndarray] = None  # explicit contents for fill == "array"

    @property
    def nbytes(self) -> int:
        return int(np.prod(self.shape, dtype=np.int64)) * ELEM_SIZE[self.dtype] if self.shape else 0


@dataclasses.dataclass
class Matrix:
    """One GEMV unit: a [M, K] matrix assembled from one or more row blocks."""

    name: str
    dtype: int
    M: int
    K: int
    parts: List[int]              # tensor indices, in row order
    scale: Optional[int] = None   # tensor index of the fp16 row scales (int8 weights)


@dataclasses.dataclass
class Checkpoint:
    workload: str
    paths: List[str]
    tensors: List[TensorSpec]
    matrices: List[Matrix]

    @property
    def data_bytes(self) -> int:
        return sum(t.nbytes for t in self.tensors)

    @property
    def weight_bytes(self) -> int:
        return sum(m.M * m.K * ELEM_SIZE[m.dtype] for m in self.matrices)

    def file_tensors(self, f: int) -> List[int]:
        return [i for i, t in enumerate(self.tensors) if t.file == f]


# --------------------------------------------------------------------------- values

def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round finite float32 values to bfloat16 bit patterns, round-to-nearest-even."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    r = (u >> 16) & 1
    r += 0x7FFF
    r += u          # finite inputs stay below 2^32
    r >>= 16
    return r.astype(np.uint16)


_BUFS: Dict[str, np.ndarray] = {}


def _buf(name: str, dtype, count: int) -> np.ndarray:
    """Per-process scratch arrays, reused across chunks (fresh pages are slow to fault in)."""
    b = _BUFS.get(name)
    if b is None or b.size < count:
        b = _BUFS[name] = np.empty(max(count, _CHUNK), dtype)
    return b[:count]


def _normal_bf16(rng, count: int, scale: float) -> np.ndarray:
    """N(0, scale) drawn in float32, rounded to bf16 (RNE), as little-endian bytes; in place."""
    v = _buf("f32", np.float32, count)
    rng.standard_normal(out=v, dtype=np.float32)
    v *= np.float32(scale)
    u = v.view(np.uint32)
    r = _buf("u32", np.uint32, count)
    np.right_shift(u, np.uint32(16), out=r)
    r &= np.uint32(1)
    r += np.uint32(0x7FFF)
    r += u
    r >>= np.uint32(16)
    o = _buf("u16", np.uint16, count)
    np.copyto(o, r, casting="unsafe")
    return o.view(np.uint8)


def _tensor_values(t: TensorSpec, start: int, count: int, rng) -> np.ndarray:
    """`count` values of `t` starting at element `start`, as raw little-endian element bytes."""
    if t.fill == "normal" and t.dtype == DT_BF16:
        return _normal_bf16(rng, count, t.scale)
    if t.fill == "ones":
        v = np.ones(count, dtype=np.float32)
    elif t.fill == "uniform":
        v = rng.uniform(-t.scale, t.scale, count).astype(np.float32)
    elif t.fill == "normal":
        v = rng.standard_normal(count, dtype=np.float32)
        v *= np.float32(t.scale)
    elif t.fill == "array":
        return np.ascontiguousarray(t.array).reshape(-1).view(np.uint8)[
            start * ELEM_SIZE[t.dtype]:(start + count) * ELEM_SIZE[t.dtype]]
    elif t.fill == "int8":
        return rng.integers(-127, 128, count, dtype=np.int8).view(np.uint8)
    elif t.fill == "rowscale":
        v = rng.uniform(t.scale, 10 * t.scale, count).astype(np.float32)
    else:
        raise ValueError(t.fill)
    if t.dtype == DT_F32:
        return v.astype("<f4").view(np.uint8)
    if t.dtype == DT_BF16:
        return f32_to_bf16_bits(v).astype("<u2").view(np.uint8)
    if t.dtype == DT_F16:
        return v.astype("<f2").view(np.uint8)
    raise ValueError("no value recipe for dtype %d" % t.dtype)


def _rng_for(t: TensorSpec, chunk: int):
    """Value stream of chunk `chunk` (of _CHUNK elements) of tensor `t`."""
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence(0, spawn_key=t.key + (chunk,))))


def make_x(K: int, dtype: int) -> np.ndarray:
    """GEMV input for inner size K: N(0,1) from PCG64(1000003 + K), cast fp64->fp32->dtype (RNE).
    int8 weights take fp16 activations, so DT_I8 returns fp16 x.

    Returned as the raw little-endian element bytes (uint8)."""
    rng = np.random.Generator(np.random.PCG64(1000003 + K))
    v = rng.standard_normal(K).astype(np.float32)
    if dtype == DT_I8:
        dtype = DT_F16
    if dtype == DT_F32:
        return v.astype("<f4").view(np.uint8).copy()
    if dtype == DT_BF16:
        return f32_to_bf16_bits(v).astype("<u2").view(np.uint8).copy()
    if dtype == DT_F16:
        return v.astype("<f2").view(np.uint8).copy()
    raise ValueError(dtype)


# --------------------------------------------------------------------------- layout / writing

def encode_index(entries: Sequence[TensorSpec]) -> bytes:
    out = [struct.pack("<I", len(entries))]
    for t in entries:
        nm = t.name.encode("utf-8")
        out.append(struct.pack("<H", len(nm)) + nm + struct.pack("<BB", t.dtype, len(t.shape)))
        out.append(struct.pack("<%dQ" % len(t.shape), *t.shape))
        out.append(struct.pack("<QQ", t.offset, t.nbytes))
    return b"".join(out)


def layout(entries: Sequence[TensorSpec]) -> Tuple[bytes, int]:
    """Assign 64-byte aligned offsets in index order; return (header+index bytes, file size)."""
    idx_len = len(encode_index(entries))  # offsets are fixed-width, so the length is known up front
    pos = -(-(16 + idx_len) // ALIGN) * ALIGN
    for t in entries:
        t.offset = pos
        pos = -(-(pos + t.nbytes) // ALIGN) * ALIGN
    idx = encode_index(entries)
    assert len(idx) == idx_len
    end = max([t.offset + t.nbytes for t in entries] + [16 + idx_len])
    return MAGIC + struct.pack("<Q", idx_len) + idx, end


def _write_chunk(path: str, t: TensorSpec, c: int) -> int:
    """Write elements [c*_CHUNK, (c+1)*_CHUNK) of `t`; each chunk draws from its own stream."""
    es = ELEM_SIZE[t.dtype]
    n = t.nbytes // es
    s = c * _CHUNK
    cnt = min(_CHUNK, n - s)
    rng = _rng_for(t, c) if t.fill in ("normal", "uniform", "int8", "rowscale") else None
    buf = np.ascontiguousarray(_tensor_values(t, s, cnt, rng))
    fd = os.open(path, os.O_WRONLY)
    try:
        os.pwrite(fd, buf, t.offset + s * es)
    finally:
        os.close(fd)
    return cnt * es


def _write_task(args):
    return _write_chunk(*args)


def write_files(ck: Checkpoint, workers: int = 0) -> Checkpoint:
    """Write every file of `ck` (headers, then blobs; blobs in parallel when workers > 1)."""
    tasks = []
    for f, path in enumerate(ck.paths):
        idxs = ck.file_tensors(f)
        entries = [ck.tensors[i] for i in idxs]
        head, size = layout(entries)
        d = os.path.dirname(path)
        if d:
            os.makedirs(d, exist_ok=True)
        with open(path, "wb") as fh:
            fh.truncate(size)
            fh.write(head)
        for i in idxs:
            t = ck.tensors[i]
            n = t.nbytes // ELEM_SIZE[t.dtype]
            tasks += [(path, t, c) for c in range(-(-n // _CHUNK))]
    if workers and workers > 1 and len(tasks) > 1:
        import multiprocessing as mp
        with mp.get_context("spawn").Pool(min(workers, len(tasks))) as pool:
            for _ in pool.imap_unordered(_write_task, tasks, chunksize=max(1, len(tasks) // (8 * workers))):
                pass
    else:
        for a in tasks:
            _write_task(a)
    return ck


# --------------------------------------------------------------------------- workloads

def tiny(outdir: str) -> Checkpoint:
    """8 fp32 256x256 matrices + 8 fp32[256] vectors in one file, U[-1,1] from PCG64(0)."""
    rng = np.random.Generator(np.random.PCG64(0))
    tensors = []
    for i in range(8):
        for nm, shape in ((f"m{i}", (256, 256)), (f"v{i}", (256,))):
            arr = rng.uniform(-1.0, 1.0, int(np.prod(shape))).astype("<f4")
            tensors.append(TensorSpec(nm, DT_F32, shape, 0, fill="array", array=arr))
    mats = [Matrix(f"m{i}", DT_F32, 256, 256, [2 * i]) for i in range(8)]
    return Checkpoint("tiny", [os.path.join(outdir, "tiny.wt")], tensors, mats)


def sweep(outdir: str, points: Sequence[int] = tuple(range(14)), rows: int = 4096) -> Checkpoint:
    """One bf16 rows x (128*2^i) matrix per file: 1 MiB ... 8 GiB at rows=4096."""
    tensors, mats, paths = [], [], []
    for f, i in enumerate(points):
        C = 128 << i
        tensors.append(TensorSpec("w", DT_BF16, (rows, C), f, key=(_STREAM_KEY["sweep"], i)))
        mats.append(Matrix(f"sweep{i}", DT_BF16, rows, C, [f]))
        paths.append(os.path.join(outdir, f"sweep_{i:02d}.wt"))
    return Checkpoint("sweep", paths, tensors, mats)


def many_shapes(n_matrices: int = 1253) -> List[Tuple[int, int]]:
    """(M, K) per matrix: half-bytes s log-uniform in [4 KiB, 4 MiB], K = 2^c (c in 5..11),
    M_half = max(1, floor(s / (2K))), M = 2 M_half.  Shape stream: SeedSequence(0).spawn(2)[0]."""
    rng = np.random.Generator(np.random.PCG64(np.random.SeedSequence(0).spawn(2)[0]))
    out = []
    for _ in range(n_matrices):
        s = math.exp(rng.uniform(math.log(4096.0), math.log(4194304.0)))
        K = 1 << int(rng.integers(5, 12))
        mh = max(1, int(s // (2 * K)))
        out.append((2 * mh, K))
    return out


def many(outdir: str, n_matrices: int = 1253) -> Checkpoint:
    """Each matrix's rows split in half across two files ("<name>#r0", "<name>#r1")."""
    tensors, mats, paths = [], [], []
    for m, (M, K) in enumerate(many_shapes(n_matrices)):
        parts = []
        for h, (r0, r1) in enumerate(((0, M // 2), (M // 2, M))):
            f = 2 * m + h
            parts.append(len(tensors))
            tensors.append(TensorSpec(f"m{m}#r{h}", DT_BF16, (r1 - r0, K), f,
                                      key=(_STREAM_KEY["many"], f)))
            paths.append(os.path.join(outdir, f"many_{f:05d}.wt"))
        mats.append(Matrix(f"m{m}", DT_BF16, M, K, parts))
    return Checkpoint("many", paths, tensors, mats)


DECODERS: Dict[str, dict] = {
    "mid": dict(layers=32, d=2560, kv=2560, ffn=6912, vocab=32000, shards=3),
    "large": dict(layers=32, d=4096, kv=1024, ffn=14336, vocab=128256, shards=4),
}


def decoder(outdir: str, which: str, layers: Optional[int] = None, shards: Optional[int] = None,
            vocab: Optional[int] = None) -> Checkpoint:
    """Decoder checkpoint in layer order: embed; per layer attn_norm, q, k, v, o, ffn_norm,
    gate, up, down; final_norm; lm_head.  Matrices are [out, in]; norms are exactly 1.0.
    Shards are filled greedily, cutting before a tensor that would pass ceil(total/shards)."""
    cfg = dict(DECODERS[which])
    if layers is not None:
        cfg["layers"] = layers
    if shards is not None:
        cfg["shards"] = shards
    if vocab is not None:
        cfg["vocab"] = vocab
    d, kv, ffn, V = cfg["d"], cfg["kv"], cfg["ffn"], cfg["vocab"]
    order: List[Tuple[str, Tuple[int, ...]]] = [("embed", (V, d))]
    for l in range(cfg["layers"]):
        p = f"layers.{l}."
        order += [(p + "attn_norm", (d,)), (p + "q", (d, d)), (p + "k", (kv, d)), (p + "v", (kv, d)),
                  (p + "o", (d, d)), (p + "ffn_norm", (d,)), (p + "gate", (ffn, d)),
                  (p + "up", (ffn, d)), (p + "down", (d, ffn))]
    order += [("final_norm", (d,)), ("lm_head", (V, d))]
    sizes = [int(np.prod(s)) * 2 for _, s in order]
    cap = -(-sum(sizes) // cfg["shards"])
    tensors, mats = [], []
    f, acc = 0, 0
    for t, ((nm, shape), sz) in enumerate(zip(order, sizes)):
        if acc > 0 and acc + sz > cap and f + 1 < cfg["shards"]:
            f, acc = f + 1, 0
        acc += sz
        if len(shape) == 1:
            tensors.append(TensorSpec(nm, DT_BF16, shape, f, fill="ones"))
        else:
            tensors.append(TensorSpec(nm, DT_BF16, shape, f, key=(_STREAM_KEY[which], t)))
            mats.append(Matrix(nm, DT_BF16, shape[0], shape[1], [t]))
    n_files = f + 1
    paths = [os.path.join(outdir, f"{which}_{s:02d}-of-{n_files:02d}.wt") for s in range(n_files)]
    return Checkpoint(which, paths, tensors, mats)


def custom(outdir: str, shapes: Sequence[Tuple[int, int]], dtype: int = DT_BF16,
           name: str = "custom", scale: float = 0.02) -> Checkpoint:
    """One file holding one [M, K] matrix per shape (edge-case and ragged-shape tests)."""
    tensors, mats = [], []
    for i, (M, K) in enumerate(shapes):
        tensors.append(TensorSpec(f"w{i}", dtype, (M, K), 0, key=(_STREAM_KEY["custom"], i),
                                  scale=scale))
        mats.append(Matrix(f"w{i}", dtype, M, K, [i]))
    return Checkpoint(name, [os.path.join(outdir, name + ".wt")], tensors, mats)


def protocol(outdir: str, matrices: int = 12, rows: int = 12288, cols: int = 3584) -> Checkpoint:
    """The paper's matched protocol by bytes (Sec. 3.1): a pass visits 12 page-cache-resident
    files of 88.1 MB each (there 12288x7168 int8 with fp16 row scales; here 12288x3584 bf16,
    the same weight bytes per file)."""
    tensors, mats, paths = [], [], []
    for f in range(matrices):
        tensors.append(TensorSpec("w", DT_BF16, (rows, cols), f, key=(_STREAM_KEY["protocol"], f)))
        mats.append(Matrix("p%d" % f, DT_BF16, rows, cols, [f]))
        paths.append(os.path.join(outdir, "protocol_%02d.wt" % f))
    return Checkpoint("protocol", paths, tensors, mats)


def protocol_q8(outdir: str, matrices: int = 12, rows: int = 12288, cols: int = 7168) -> Checkpoint:
    """The paper's matched protocol (Sec. 3.1): 12 files, each one int8 rows x cols matrix "w"
    (88.1 MB at 12288x7168) and its fp16 row scales "w.scale"."""
    tensors, mats, paths = [], [], []
    for f in range(matrices):
        tensors.append(TensorSpec("w", DT_I8, (rows, cols), f, fill="int8", key=(_STREAM_KEY["protocol_q8"], 2 * f)))
        tensors.append(TensorSpec("w.scale", DT_F16, (rows,), f, fill="rowscale", scale=0.002,
                                  key=(_STREAM_KEY["protocol_q8"], 2 * f + 1)))
        mats.append(Matrix("p%d" % f, DT_I8, rows, cols, [2 * f], scale=2 * f + 1))
        paths.append(os.path.join(outdir, "protocol_q8_%02d.wt" % f))
    return Checkpoint("protocol_q8", paths, tensors, mats)


def custom_q8(outdir: str, shapes: Sequence[Tuple[int, int]], name: str = "custom_q8") -> Checkpoint:
    """One file holding, per shape, an int8 [M, K] matrix "w<i>" and its fp16 scales "w<i>.scale"."""
    tensors, mats = [], []
    for i, (M, K) in enumerate(shapes):
        tensors.append(TensorSpec(f"w{i}", DT_I8, (M, K), 0, fill="int8", key=(_STREAM_KEY["custom"], 1000 + 2 * i)))
        tensors.append(TensorSpec(f"w{i}.scale", DT_F16, (M,), 0, fill="rowscale", scale=0.002,
                                  key=(_STREAM_KEY["custom"], 1001 + 2 * i)))
        mats.append(Matrix(f"w{i}", DT_I8, M, K, [2 * i], scale=2 * i + 1))
    return Checkpoint(name, [os.path.join(outdir, name + ".wt")], tensors, mats)


def build(workload: str, outdir: str, workers: int = 0, **kw) -> Checkpoint:
    """Describe and write a workload; returns the Checkpoint (paths, tensors, matrices)."""
    if workload == "tiny":
        ck = tiny(outdir)
    elif workload == "protocol":
        ck = protocol(outdir, **kw)
    elif workload == "protocol_q8":
        ck = protocol_q8(outdir, **kw)
    elif workload == "sweep":
        ck = sweep(outdir, **kw)
    elif workload == "many":
        ck = many(outdir, **kw)
    elif workload in DECODERS:
        ck = decoder(outdir, workload, **kw)
    else:
        raise ValueError(workload)
    return write_files(ck, workers=workers)
