"""Pins of the oracle's INT8 storage of the factors (Sec. 5.3, Table 2:
asymmetric INT8 quantisation on top of the low-rank cache), against what the
definition and arithmetic fix rather than against itself:

- a worked group whose step, codes and read-back values were derived by hand
  (tests/golden/int8_group_hand_example.json);
- values on an exact grid of the step (read back bit-exactly);
- brute force: every code is the nearest of all 256 (exact rational check);
- the error bound |x - x^| <= s/2 + bf16 rounding, and the step's bounds;
- special cases: constant groups, signed zeros, the padding of edge tiles;
- the stored bytes behind Table 2's doubling of the KV reduction."""
import json
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import milo_int8 as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "int8_group_hand_example.json")


def bits_of(x):
    """float values (exact in bf16) -> bf16 bits."""
    a = np.asarray(x, dtype=np.float32)
    u = a.view(np.uint32)
    assert np.all((u & 0xFFFF) == 0), "value not exact in bf16"
    return (u >> 16).astype(np.uint16)


def f64(bits):
    return Q.bf16_to_f32(bits).astype(np.float64)


def random_group(rng, scale=1.0, shift=0.0):
    x = (rng.standard_normal(64) * scale + shift).astype(np.float32)
    return Q.f32_to_bf16_rne(x)


def test_hand_example():
    g = json.load(open(GOLDEN))
    vals = np.array(g["values"])
    idx = (np.arange(8)[:, None] + np.arange(8)[None, :]) % 8
    tile = bits_of(vals[idx])
    codes, m, s = Q.quantize_group(tile)
    assert m == g["m_bits"] and s == g["s_bits"]
    assert f64(np.uint16(s))[()] == g["s"]
    assert np.array_equal(codes, np.array(g["codes"], dtype=np.uint8)[idx])
    back = f64(Q.dequantize_group(codes, m, s))
    assert np.array_equal(back, np.array(g["read_back"])[idx])


@pytest.mark.parametrize("k", [-12, -3, 0, 4])
def test_exact_grid_reads_back_exactly(k):
    """Values (c - 128) 2^k with c over [0, 255] (both ends present): the step
    is exactly 2^k, the codes are c, and the read-back is the input."""
    rng = np.random.default_rng(k + 100)
    c = rng.integers(0, 256, size=64)
    c[3], c[40] = 0, 255
    x = ((c - 128) * 2.0 ** k).astype(np.float32)
    codes, m, s = Q.quantize_group(bits_of(x))
    assert f64(np.uint16(s))[()] == 2.0 ** k
    assert f64(np.uint16(m))[()] == -128 * 2.0 ** k
    assert np.array_equal(codes.astype(np.int64), c)
    assert np.array_equal(Q.dequantize_group(codes, m, s), bits_of(x))


def exact_q(m_bits, s_bits):
    return Fraction(float(f64(np.uint16(m_bits))[()])), Fraction(float(f64(np.uint16(s_bits))[()]))


@pytest.mark.parametrize("seed", range(6))
def test_codes_are_nearest_by_brute_force(seed):
    """Over all 256 codes, the chosen one minimises |x - (m + s c)| in exact
    arithmetic, up to fp32 rounding of the decision (a near-tie may go either
    way by one part in 2^20 of the step)."""
    rng = np.random.default_rng(seed)
    scale = 10.0 ** rng.uniform(-4, 3)
    x_bits = random_group(rng, scale, shift=rng.uniform(-2, 2) * scale)
    codes, m_bits, s_bits = Q.quantize_group(x_bits)
    m, s = exact_q(m_bits, s_bits)
    xs = [Fraction(float(v)) for v in f64(x_bits)]
    tol = s / (1 << 20)
    for x, c in zip(xs, codes.astype(int)):
        best = min(abs(x - (m + s * k)) for k in range(256))
        assert abs(x - (m + s * c)) <= best + tol


@pytest.mark.parametrize("seed", range(8))
def test_error_bound_and_step_bounds(seed):
    rng = np.random.default_rng(1000 + seed)
    scale = 10.0 ** rng.uniform(-6, 4)
    x_bits = random_group(rng, scale)
    codes, m_bits, s_bits = Q.quantize_group(x_bits)
    x = f64(x_bits)
    m, s = f64(np.uint16(m_bits))[()], f64(np.uint16(s_bits))[()]
    span = x.max() - x.min()
    # step: at least span / 255, at most that rounded up to 8 significant bits
    assert s * 255 >= span * (1 - 2.0 ** -23)
    assert s <= span / 255 * (1 + 2.0 ** -7) * (1 + 2.0 ** -23)
    assert m == x.min()
    # the minimum reads back exactly; the largest code is at least 254
    assert codes.reshape(-1)[np.argmin(x)] == 0
    assert codes.max() >= 254
    back = f64(Q.dequantize_group(codes, m_bits, s_bits))
    bound = s / 2 * (1 + 2.0 ** -20) + 2.0 ** -8 * np.abs(back)
    assert np.all(np.abs(x - back) <= bound)


def test_constant_zero_and_signed_zero_groups():
    for v in (0.0, 3.25, -7.5):
        x = bits_of(np.full(64, v))
        codes, m, s = Q.quantize_group(x)
        assert s == 0 and not codes.any()
        assert np.array_equal(Q.dequantize_group(codes, m, s), x)
    # -0 and +0 mixed: the stored minimum is +0 whichever zero is smallest
    z = np.zeros(64, dtype=np.uint16)
    z[::3] = 0x8000
    codes, m, s = Q.quantize_group(z)
    assert m == 0 and s == 0 and not codes.any()
    assert not Q.dequantize_group(codes, m, s).any()


def test_tiles_pad_edges_with_zero():
    """A 5 x 11 factor: two tiles, padded with zeros that take part in the
    group's minimum and maximum (all values positive here, so m = 0 for
    every tile); the read-back drops the padding."""
    rng = np.random.default_rng(7)
    F = (1.0 + rng.random((5, 11))).astype(np.float32)
    Fb = Q.f32_to_bf16_rne(F)
    T = Q.tiles(Fb, 5, 11)
    assert T.shape == (1, 2, 8, 8)
    assert np.array_equal(T[0, 1, :5, :3], Fb[:, 8:])
    assert not T[0, 1, 5:].any() and not T[0, 1, :, 3:].any()
    codes, m, s = Q.quantize_matrix(Fb, 5, 11)
    assert codes.shape == (1, 2, 8, 8) and not m.any()
    for j in range(2):
        c2, m2, s2 = Q.quantize_group(T[0, j])
        assert np.array_equal(codes[0, j], c2) and m[0, j] == m2 and s[0, j] == s2
    back = Q.dequantize_matrix(codes, m, s, 5, 11)
    assert back.shape == (5, 11)
    step = f64(s).max()
    assert np.abs(f64(back) - f64(Fb)).max() <= step / 2 + 2.0 ** -8 * 2.0


def test_reciprocal_overflow_gives_code_zero():
    """A span so small that 1/s overflows fp32: every code 0, read back m."""
    x = np.zeros(64, dtype=np.uint16)
    x[5] = 0x0001           # the smallest bf16 subnormal, 2^-133
    codes, m, s = Q.quantize_group(x)
    assert m == 0 and s == 0x0001 and not codes.any()


def test_stored_bytes_double_the_reduction():
    """Table 2: INT8 on top of MILO doubles the KV reduction (2x -> 4x).  The
    codes alone are exactly half of the bf16 tiles; with the two bf16
    parameters per 64-value group the factor is 128/68."""
    for rows, cols in ((512, 128), (37, 96), (8, 8), (1, 1)):
        b16, b8 = Q.stored_bytes(rows, cols)
        ntiles = b16 // 128
        assert b8 - 4 * ntiles == b16 // 2
        assert Fraction(b16, b8) == Fraction(128, 68)


def test_matrix_form_is_the_group_rule_tile_by_tile():
    """quantize_matrix / dequantize_matrix apply the one-group rule to every
    tile (checked tile by tile against quantize_group / dequantize_group)."""
    rng = np.random.default_rng(11)
    rows, cols = 37, 21
    F = (rng.standard_normal((rows, cols)) * np.logspace(0, -3, cols)[None, :]).astype(np.float32)
    Fb = Q.f32_to_bf16_rne(F)
    codes, m, s = Q.quantize_matrix(Fb, rows, cols)
    T = Q.tiles(Fb, rows, cols)
    back = Q.dequantize_matrix(codes, m, s, rows, cols)
    for i in range(T.shape[0]):
        for j in range(T.shape[1]):
            c1, m1, s1 = Q.quantize_group(T[i, j])
            assert np.array_equal(codes[i, j], c1) and m[i, j] == m1 and s[i, j] == s1
            d1 = Q.dequantize_group(c1, m1, s1)
            r0, c0 = 8 * i, 8 * j
            blk = back[r0:r0 + 8, c0:c0 + 8]
            assert np.array_equal(blk, d1[:blk.shape[0], :blk.shape[1]])
