"""The arithmetic the parallel second level of the tree digest rests on, restated on the
host and checked against the oracle's literal FNV-1a-64 (no GPU): a chain over a byte
stream cut into chunks, combined from per-chunk low-byte tables, a low-word run from each
chunk's starting low byte, a scan of the low word and a fold of the high word, equals the
serial chain.  A wrong derivation (a dropped d term, the high word's carry, the wrong power
of p, the packed 16-bit lanes) fails here before any kernel runs."""
import struct

import numpy as np
import pytest

import oracle

M32 = 0xFFFFFFFF
P = 0x1B3  # FNV-1a-64's prime is 2^40 + 0x1b3


def step(lo, hi, b):
    """One byte on the split state: x = lo ^ b; x p = low32(x 0x1b3) + (hi 0x1b3 + (x << 8) +
    high32(x 0x1b3)) 2^32 mod 2^64."""
    x = lo ^ b
    w = x * P
    return w & M32, (hi * P + (w >> 32) + (x << 8)) & M32


def run(lo, hi, data):
    for b in data:
        lo, hi = step(lo, hi, b)
    return lo, hi


def low_byte_table(chunk):
    """l_end for all 256 starting low bytes, four starts per 'thread' in two registers of two
    16-bit lanes, multiplier 0xb3 (= p mod 256); the mask of one step merged into the next."""
    mask = 0x00FF00FF
    out = [0] * 256
    for tid in range(64):
        r0 = tid | (tid + 64) << 16
        r1 = (tid + 128) | (tid + 192) << 16
        for b in chunk:
            bb = b | b << 16
            r0 = (((r0 & mask) ^ bb) * 0xB3) & M32
            r1 = (((r1 & mask) ^ bb) * 0xB3) & M32
        out[tid], out[tid + 64] = r0 & 0xFF, (r0 >> 16) & 0xFF
        out[tid + 128], out[tid + 192] = r1 & 0xFF, (r1 >> 16) & 0xFF
    return out


def chunked(head, stream, m):
    """FNV-1a-64 of head + stream with the stream cut into chunks of m bytes."""
    lo, hi = run(0x84222325, 0xCBF29CE4, head)
    chunks = [stream[i:i + m] for i in range(0, len(stream), m)]
    tabs = [low_byte_table(c) for c in chunks]
    ls, l = [], lo & 0xFF                       # walk the low byte through the tables
    for t in tabs:
        ls.append(l)
        l = t[l]
    bparts = []                                 # B from the starting low byte alone
    for c, l0 in zip(chunks, ls):
        lo_end = l0
        for b in c:
            lo_end = ((lo_end ^ b) * P) & M32
        bparts.append((lo_end - pow(P, len(c), 1 << 32) * l0) & M32)
    starts = []                                 # lo at every chunk start
    for c, bp in zip(chunks, bparts):
        starts.append(lo)
        lo = (pow(P, len(c), 1 << 32) * lo + bp) & M32
    for c, s, l0 in zip(chunks, starts, ls):    # the walk saw the true low bytes
        assert s & 0xFF == l0
    for c, s in zip(chunks, starts):            # hi folded over H from each true start
        _, h = run(s, 0, c)
        hi = (pow(P, len(c), 1 << 32) * hi + h) & M32
    return hi << 32 | lo


@pytest.mark.parametrize("nwords,m", [(1, 8), (2, 8), (5, 16), (9, 24), (40, 64), (64, 512)])
def test_chunked_chain_equals_the_serial_digest(nwords, m):
    rng = np.random.default_rng(nwords * 1000 + m)
    for trial in range(4):
        words = rng.integers(0, 2 ** 63, nwords, dtype=np.uint64) * (1 + trial % 2)
        if trial == 2:
            words[:] = 0
        if trial == 3:
            words[:] = np.uint64(2 ** 64 - 1)
        n = int(rng.integers(0, 2 ** 40))
        head = struct.pack("<Q", n)
        stream = words.astype("<u8").tobytes()
        assert chunked(head, stream, m) == oracle.fnv1a64(head + stream)


def test_chunked_chain_over_real_leaf_digests():
    """The second level proper: the stream is LE64 of the 4096-byte leaf digests."""
    rng = np.random.default_rng(3)
    data = rng.integers(0, 256, 4096 * 37 + 11, dtype=np.uint8)
    leaves = [oracle.fnv1a64(data[i:i + 4096]) for i in range(0, data.size, 4096)]
    stream = struct.pack("<%dQ" % len(leaves), *leaves)
    assert chunked(struct.pack("<Q", data.size), stream, 8 * 5) == oracle.fnv_tree(data)
