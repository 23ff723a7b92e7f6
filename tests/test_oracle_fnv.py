"""Pins for the oracle's byte digests (D_plain, D_tree), independent of the oracle itself.

D_plain is FNV-1a-64; D_tree is FNV-1a-64 over LE64(n) and the LE64 digests of
4096-byte leaves (the reading of "per-tensor 64-bit FNV-1a" that lets a GPU
hash large tensors in parallel).
"""
import struct

import numpy as np
import pytest

import oracle

M64 = (1 << 64) - 1
# FNV prime for 64 bits, as the FNV specification states it: 2^40 + 2^8 + 0xb3
PRIME = (1 << 40) + (1 << 8) + 0xB3


def test_offset_basis_rederived_from_spec_construction():
    # The FNV specification defines the 64-bit offset basis as the FNV-0 hash
    # (basis 0, multiply then xor) of its author's signature line.  Deriving it
    # here pins both the oracle's basis and, through it, its prime.
    sig = b"chongo <Landon Curt Noll> /\\../\\"
    h = 0
    for b in sig:
        h = (h * PRIME) & M64
        h ^= b
    assert oracle.fnv1a64(b"") == h


@pytest.mark.parametrize("n", [1, 2, 7, 64, 1000, 4096, 4097])
def test_step_inversion_recovers_basis(n):
    # FNV-1a is xor-then-multiply by an odd prime; undoing each step with the
    # prime's inverse mod 2^64 must walk back to the basis.  A wrong prime, a
    # swapped step order (FNV-1) or a skipped byte all break this.
    rng = np.random.default_rng(n)
    data = rng.integers(0, 256, n, dtype=np.uint8)
    h = oracle.fnv1a64(data)
    inv = pow(PRIME, -1, 1 << 64)
    for b in data[::-1]:
        h = (h * inv) & M64
        h ^= int(b)
    assert h == oracle.fnv1a64(b"")


def test_single_byte_closed_form():
    basis = oracle.fnv1a64(b"")
    for b in (0, 1, 0x7F, 0x80, 0xFF):
        assert oracle.fnv1a64(bytes([b])) == ((basis ^ b) * PRIME) & M64


def _le64(v):
    return struct.pack("<Q", v)


@pytest.mark.parametrize("n", [0, 1, 100, 4095, 4096])
def test_tree_equals_plain_of_header_and_one_leaf(n):
    data = np.random.default_rng(10 + n).integers(0, 256, n, dtype=np.uint8).tobytes()
    expect = oracle.fnv1a64(_le64(n) + (_le64(oracle.fnv1a64(data)) if n else b""))
    assert oracle.fnv_tree(data) == expect


@pytest.mark.parametrize("n", [4097, 8192, 3 * 4096 + 17, 10 * 4096])
def test_tree_leaf_boundaries(n):
    data = np.random.default_rng(n).integers(0, 256, n, dtype=np.uint8).tobytes()
    leaves = [oracle.fnv1a64(data[s:s + 4096]) for s in range(0, n, 4096)]
    expect = oracle.fnv1a64(_le64(n) + b"".join(_le64(l) for l in leaves))
    assert oracle.fnv_tree(data) == expect


def test_digests_see_every_byte():
    rng = np.random.default_rng(3)
    data = bytearray(rng.integers(0, 256, 3 * 4096 + 5, dtype=np.uint8).tobytes())
    base_p, base_t = oracle.fnv1a64(bytes(data)), oracle.fnv_tree(bytes(data))
    for pos in (0, 4095, 4096, 8191, len(data) - 1):
        d2 = bytearray(data)
        d2[pos] ^= 0x01
        assert oracle.fnv1a64(bytes(d2)) != base_p
        assert oracle.fnv_tree(bytes(d2)) != base_t
    # length is part of the tree digest: a trailing zero byte changes it
    assert oracle.fnv_tree(bytes(data) + b"\0") != base_t


def test_numpy_and_bytes_inputs_agree():
    data = np.arange(5000, dtype=np.uint16)
    assert oracle.fnv1a64(data) == oracle.fnv1a64(data.tobytes())
    assert oracle.fnv_tree(data) == oracle.fnv_tree(data.tobytes())
