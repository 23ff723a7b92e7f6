"""Pins for the oracle's fp64 GEMV (y = W x, W [M, K] row-major [out, in]).

Checks come from outside the oracle: exact integer arithmetic, element decodes
through ``struct``/numpy's own half type, and numpy's float64 matmul.
"""
import math
import struct
from fractions import Fraction

import numpy as np
import pytest

import oracle
from paper_2608_12114_gb300 import synth

F32, BF16, F16 = synth.DT_F32, synth.DT_BF16, synth.DT_F16


def enc(vals, dtype):
    """Encode exactly-representable values as raw element bytes (via struct / numpy)."""
    v = np.asarray(vals, np.float64)
    if dtype == F32:
        return np.frombuffer(struct.pack("<%df" % v.size, *v.ravel()), np.uint8).copy()
    if dtype == BF16:
        raw = struct.pack("<%df" % v.size, *v.ravel())
        hi = [raw[4 * i + 2:4 * i + 4] for i in range(v.size)]
        assert all(raw[4 * i:4 * i + 2] == b"\0\0" for i in range(v.size)), "not exact in bf16"
        return np.frombuffer(b"".join(hi), np.uint8).copy()
    if dtype == F16:
        h = v.astype(np.float16)
        assert np.all(h.astype(np.float64) == v), "not exact in f16"
        return h.astype("<f2").view(np.uint8).copy()
    raise ValueError(dtype)


@pytest.mark.parametrize("dtype", [F32, BF16, F16])
def test_integer_matrix_exact(dtype):
    rng = np.random.default_rng(1)
    M, K = 13, 37
    W = rng.integers(-8, 9, (M, K))
    x = rng.integers(-4, 5, K)
    yhat, a = oracle.gemv(enc(W, dtype), dtype, M, K, enc(x, dtype))
    for i in range(M):
        assert yhat[i] == sum(int(W[i, j]) * int(x[j]) for j in range(K))
        assert a[i] == sum(abs(int(W[i, j]) * int(x[j])) for j in range(K))


@pytest.mark.parametrize("dtype", [F32, BF16])
def test_one_hot_returns_column(dtype):
    rng = np.random.default_rng(2)
    M, K = 9, 16
    if dtype == BF16:
        Wb = synth.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32))
        Wraw = Wb.astype("<u2").view(np.uint8)
        Wval = np.array([struct.unpack("<f", b"\0\0" + struct.pack("<H", int(u)))[0]
                         for u in Wb.ravel()]).reshape(M, K)
    else:
        Wv = rng.standard_normal((M, K)).astype(np.float32)
        Wraw = Wv.astype("<f4").view(np.uint8)
        Wval = Wv.astype(np.float64)
    for j in (0, 5, K - 1):
        x = np.zeros(K)
        x[j] = 1.0
        yhat, _ = oracle.gemv(Wraw, dtype, M, K, enc(x, dtype))
        assert np.array_equal(yhat, Wval[:, j])  # W[:, j]: orientation is [out, in]


def test_ones_gives_row_sums_and_zero_gives_zero():
    rng = np.random.default_rng(3)
    M, K = 7, 300
    Wv = rng.standard_normal((M, K)).astype(np.float32)
    raw = Wv.astype("<f4").view(np.uint8)
    yhat, a = oracle.gemv(raw, F32, M, K, enc(np.ones(K), F32))
    for i in range(M):
        exact = sum(Fraction(float(w)) for w in Wv[i])
        assert abs(Fraction(yhat[i]) - exact) <= Fraction(K) * Fraction(2) ** -52 * abs(Fraction(a[i]))
        assert a[i] == pytest.approx(math.fsum(abs(float(w)) for w in Wv[i]), rel=1e-15)
    y0, a0 = oracle.gemv(raw, F32, M, K, enc(np.zeros(K), F32))
    assert not y0.any() and not a0.any()


def test_matches_numpy_float64():
    rng = np.random.default_rng(4)
    M, K = 64, 1000
    Wv = rng.standard_normal((M, K)).astype(np.float32)
    xv = rng.standard_normal(K).astype(np.float32)
    yhat, a = oracle.gemv(Wv.view(np.uint8), F32, M, K, xv.view(np.uint8))
    ref = Wv.astype(np.float64) @ xv.astype(np.float64)
    refa = np.abs(Wv.astype(np.float64) * xv.astype(np.float64)).sum(1)
    assert np.allclose(yhat, ref, rtol=0, atol=1e-12 * refa.max())
    assert np.allclose(a, refa, rtol=1e-13)


def test_bf16_decode_special_patterns():
    # bf16 is the top half of an IEEE single: decode through struct, not the oracle
    pats = [0x3F80, 0xC000, 0x0001, 0x8001, 0x7F7F, 0x0080, 0x0000, 0x8000, 0x3E4D]
    W = np.array(pats, "<u2").view(np.uint8)
    one = np.array([0x3F80], "<u2").view(np.uint8)
    yhat, _ = oracle.gemv(W, BF16, len(pats), 1, one)
    want = [struct.unpack("<f", struct.pack("<I", p << 16))[0] for p in pats]
    assert list(yhat) == want
    assert want[2] == 2.0 ** -133 and want[1] == -2.0


def test_f16_decode_all_finite_patterns():
    bits = np.arange(1 << 16, dtype=np.uint16)
    vals = bits.view(np.float16)
    keep = np.isfinite(vals)
    W = bits[keep].astype("<u2").view(np.uint8)
    one = np.array([1.0], "<f2").view(np.uint8)
    yhat, _ = oracle.gemv(W, F16, int(keep.sum()), 1, one)
    assert np.array_equal(yhat, vals[keep].astype(np.float64))


def test_rows_subset_matches_full():
    rng = np.random.default_rng(5)
    M, K = 50, 96
    Wb = synth.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32)).view(np.uint8)
    x = synth.make_x(K, BF16)
    y, a = oracle.gemv(Wb, BF16, M, K, x)
    rows = [0, 17, 49, 3]
    ys, as_ = oracle.gemv_rows(Wb, BF16, M, K, x, rows)
    assert np.array_equal(ys, y[rows]) and np.array_equal(as_, a[rows])
    with pytest.raises(oracle.OracleError):
        oracle.gemv_rows(Wb, BF16, M, K, x, [M])


def test_error_metric():
    yhat = np.array([1.0, -2.0, 0.0])
    a = np.array([2.0, 4.0, 0.0])
    assert oracle.gemv_error(np.array([1.0, -2.0, 0.0]), yhat, a) == 0.0
    assert oracle.gemv_error(np.array([1.002, -2.0, 0.0]), yhat, a) == pytest.approx(1e-3)
    assert oracle.gemv_error(np.array([1.0, -2.0, 1e-30]), yhat, a) == float("inf")


def test_empty_shapes():
    y, a = oracle.gemv(np.zeros(0, np.uint8), BF16, 0, 16, synth.make_x(16, BF16))
    assert y.size == 0
    y, a = oracle.gemv(np.zeros(0, np.uint8), BF16, 4, 0, np.zeros(0, np.uint8))
    assert not y.any() and not a.any()


# ----------------------------------------------------------------------------- int8 + fp16 row scales

def _f16(v):
    return np.asarray(v, np.float16).astype("<f2").view(np.uint8)


def test_q8_integer_exact_with_power_of_two_scales():
    rng = np.random.default_rng(11)
    M, K = 11, 53
    W = rng.integers(-128, 128, (M, K)).astype(np.int8)
    x = rng.integers(-3, 4, K)
    s = 2.0 ** rng.integers(-6, 2, M)
    yhat, a = oracle.gemv_q8(W.view(np.uint8), _f16(s), M, K, _f16(x))
    for i in range(M):
        exact = sum(int(W[i, j]) * int(x[j]) for j in range(K))
        assert yhat[i] == s[i] * exact
        assert a[i] == abs(s[i]) * sum(abs(int(W[i, j]) * int(x[j])) for j in range(K))


def test_q8_one_hot_gives_scaled_column_and_matches_numpy():
    rng = np.random.default_rng(12)
    M, K = 40, 96
    W = rng.integers(-128, 128, (M, K)).astype(np.int8)
    s = rng.uniform(0.001, 0.02, M).astype(np.float16)
    for j in (0, 17, K - 1):
        x = np.zeros(K, np.float16)
        x[j] = 1.0
        yhat, _ = oracle.gemv_q8(W.view(np.uint8), s.view(np.uint8), M, K, x.view(np.uint8))
        assert np.array_equal(yhat, s.astype(np.float64) * W[:, j].astype(np.float64))
    xv = rng.standard_normal(K).astype(np.float16)
    yhat, a = oracle.gemv_q8(W.view(np.uint8), s.view(np.uint8), M, K, xv.view(np.uint8))
    ref = s.astype(np.float64) * (W.astype(np.float64) @ xv.astype(np.float64))
    assert np.allclose(yhat, ref, rtol=1e-12, atol=0)
    yr, ar = oracle.gemv_q8(W.view(np.uint8), s.view(np.uint8), M, K, xv.view(np.uint8), rows=[5, 0, 39])
    assert list(yr) == [yhat[5], yhat[0], yhat[39]] and list(ar) == [a[5], a[0], a[39]]
    with pytest.raises(oracle.OracleError):
        oracle.gemv_q8(W.view(np.uint8), s.view(np.uint8), M, K, xv.view(np.uint8), rows=[M])


# ----------------------------------------------------------------------------- T activation columns

@pytest.mark.parametrize("T", [1, 5, 8, 9, 16])
def test_cols_integer_exact_and_orientation(T):
    """X is [T, K] row-major: column t of the result uses row t of X.  Distinct integer
    columns make a transposed or shared X fail.  T spans one column, both sides of the
    8-column tile boundary and the largest T."""
    rng = np.random.default_rng(31 + T)
    M, K = 6, 40
    W = rng.integers(-8, 9, (M, K))
    X = rng.integers(-4, 5, (T, K))
    Y, A = oracle.gemv_cols(enc(W, BF16), BF16, M, K, enc(X, BF16), T)
    assert Y.shape == (T, M)
    for t in range(T):
        for i in range(M):
            assert Y[t, i] == sum(int(W[i, j]) * int(X[t, j]) for j in range(K))
            assert A[t, i] == sum(abs(int(W[i, j]) * int(X[t, j])) for j in range(K))


def test_cols_int8_scaled_exact_and_matches_numpy():
    rng = np.random.default_rng(32)
    M, K, T = 9, 64, 3
    W = rng.integers(-128, 128, (M, K)).astype(np.int8)
    X = rng.integers(-3, 4, (T, K))
    s = 2.0 ** rng.integers(-5, 2, M)
    Y, _ = oracle.gemv_cols(W.view(np.uint8), 3, M, K, _f16(X), T, scale=_f16(s))
    for t in range(T):
        for i in range(M):
            assert Y[t, i] == s[i] * sum(int(W[i, j]) * int(X[t, j]) for j in range(K))
    Xf = rng.standard_normal((T, K)).astype(np.float16)
    sf = rng.uniform(0.001, 0.02, M).astype(np.float16)
    Y, _ = oracle.gemv_cols(W.view(np.uint8), 3, M, K, Xf.view(np.uint8), T, scale=sf.view(np.uint8))
    ref = (W.astype(np.float64) @ Xf.astype(np.float64).T).T * sf.astype(np.float64)[None, :]
    assert np.allclose(Y, ref, rtol=1e-12, atol=0)


def test_cols_rows_subset_and_single_column():
    rng = np.random.default_rng(33)
    M, K, T = 20, 48, 4
    Wb = synth.f32_to_bf16_bits(rng.standard_normal((M, K)).astype(np.float32)).view(np.uint8)
    X = synth.f32_to_bf16_bits(rng.standard_normal((T, K)).astype(np.float32)).view(np.uint8)
    Y, A = oracle.gemv_cols(Wb, BF16, M, K, X, T)
    Ys, As = oracle.gemv_cols(Wb, BF16, M, K, X, T, rows=[3, 19, 0])
    assert np.array_equal(Ys, Y[:, [3, 19, 0]]) and np.array_equal(As, A[:, [3, 19, 0]])
    y1, a1 = oracle.gemv(Wb, BF16, M, K, X.reshape(T, -1)[2])
    assert np.array_equal(Y[2], y1) and np.array_equal(A[2], a1)
    with pytest.raises(oracle.OracleError):
        oracle.gemv_cols(Wb, BF16, M, K, X[:-2], T)
