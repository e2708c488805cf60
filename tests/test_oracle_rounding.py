"""Pins for the oracle's storage rounding (Sec. 3.2-3.3; factors are rounded
individually, remark after Thm 4.1).

The oracle converts binary64 to binary32/binary16 from the IEEE 754
definition with integer operations.  It is pinned here against facts that do
not come from the oracle: numpy's and CPython's direct conversions, the
exhaustive set of binary16 values and the midpoints between them, and the
format's closed-form thresholds.
"""
import struct

import numpy as np
import pytest

import oracle


def f16_via_numpy(x):
    with np.errstate(over="ignore"):
        return np.asarray(x, dtype=np.float64).astype(np.float16).view(np.uint16)


def f32_via_numpy(x):
    with np.errstate(over="ignore"):
        return np.asarray(x, dtype=np.float64).astype(np.float32).view(np.uint32)


def test_direct_conversion_not_double_rounding():
    # 1 + 2^-11 + 2^-40 lies just above the midpoint between 1 and 1 + 2^-10:
    # direct rounding gives 1 + 2^-10; rounding via binary32 first would give a
    # tie that rounds to even (1.0).
    x = 1.0 + 2.0 ** -11 + 2.0 ** -40
    assert oracle.round_bits(np.array([x]), "f16")[0] == 0x3C01
    assert struct.unpack("<H", struct.pack("<e", x))[0] == 0x3C01


def test_exhaustive_binary16_values_roundtrip():
    allbits = np.arange(65536, dtype=np.uint16)
    vals = allbits.view(np.float16).astype(np.float64)
    finite = np.isfinite(vals)
    got = oracle.round_bits(vals[finite], "f16")
    assert np.array_equal(got, allbits[finite])
    # decode agrees with numpy's widening for every pattern (NaN-aware)
    dec = oracle.decode(allbits, "f16")
    assert np.array_equal(np.isnan(dec), np.isnan(vals))
    ok = ~np.isnan(vals)
    assert np.array_equal(dec[ok], vals[ok])


def test_binary16_midpoints_ties_to_even():
    pos = np.arange(0, 0x7C00, dtype=np.uint16)          # +0 .. max finite
    lo = pos[:-1].view(np.float16).astype(np.float64)
    hi = pos[1:].view(np.float16).astype(np.float64)
    mid = (lo + hi) / 2.0                                   # exact in binary64
    got = oracle.round_bits(mid, "f16")
    even = np.where(pos[:-1] % 2 == 0, pos[:-1], pos[1:])
    assert np.array_equal(got, even)
    up = np.nextafter(mid, np.inf)
    dn = np.nextafter(mid, -np.inf)
    assert np.array_equal(oracle.round_bits(up, "f16"), pos[1:])
    assert np.array_equal(oracle.round_bits(dn, "f16"), pos[:-1])
    # and the negative half-line mirrors it
    assert np.array_equal(oracle.round_bits(-mid, "f16"), even | 0x8000)


def test_binary16_special_values_and_thresholds():
    cases = [
        (0.0, 0x0000), (-0.0, 0x8000), (np.inf, 0x7C00), (-np.inf, 0xFC00),
        (65504.0, 0x7BFF),                    # largest finite half
        (65519.999999, 0x7BFF),               # below the overflow midpoint
        (65520.0, 0x7C00),                    # midpoint to 2^16 ties to even -> inf
        (-65520.0, 0xFC00),
        (2.0 ** -24, 0x0001),                 # smallest subnormal
        (2.0 ** -25, 0x0000),                 # half of it: tie to even -> 0
        (np.nextafter(2.0 ** -25, 1.0), 0x0001),
        (1.5 * 2.0 ** -24, 0x0002),           # tie between 1 and 2 quanta -> 2
        (2.5 * 2.0 ** -24, 0x0002),           # tie between 2 and 3 quanta -> 2
        (2.0 ** -14, 0x0400),                 # smallest normal
        ((2.0 ** -14) - 2.0 ** -25, 0x0400),  # tie between max subnormal and min normal -> even
        (5e-324, 0x0000),                     # binary64 subnormal
        (-5e-324, 0x8000),
        (1e300, 0x7C00),
    ]
    for x, want in cases:
        assert int(oracle.round_bits(np.array([x]), "f16")[0]) == want, x
    nan = oracle.round_bits(np.array([np.nan, -np.nan]), "f16")
    assert np.all((nan & 0x7C00) == 0x7C00) and np.all((nan & 0x03FF) != 0)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_random_doubles_match_numpy_and_cpython(seed):
    rng = np.random.default_rng(seed)
    # wide exponent spread: subnormal, normal and overflowing magnitudes
    x = rng.standard_normal(200_000) * np.exp2(rng.uniform(-30, 20, 200_000))
    x[:1000] = rng.standard_normal(1000)        # typical factor magnitudes
    assert np.array_equal(oracle.round_bits(x, "f16"), f16_via_numpy(x))
    y = rng.standard_normal(200_000) * np.exp2(rng.uniform(-160, 140, 200_000))
    assert np.array_equal(oracle.round_bits(y, "f32"), f32_via_numpy(y))
    py16 = np.array([struct.unpack("<H", struct.pack("<e", v))[0] for v in x[:2000]
                     if abs(v) < 65504.0], dtype=np.uint16)
    x_ok = np.array([v for v in x[:2000] if abs(v) < 65504.0])
    assert np.array_equal(oracle.round_bits(x_ok, "f16"), py16)
    py32 = np.array([struct.unpack("<I", struct.pack("<f", v))[0] for v in y[:2000]
                     if abs(v) < 3.4e38], dtype=np.uint32)
    y_ok = np.array([v for v in y[:2000] if abs(v) < 3.4e38])
    assert np.array_equal(oracle.round_bits(y_ok, "f32"), py32)


def test_binary32_thresholds():
    fmax = float(np.finfo(np.float32).max)
    ulp = 2.0 ** (127 - 23)
    cases = [
        (fmax, 0x7F7FFFFF),
        (fmax + ulp / 2, 0x7F800000),                       # tie -> even -> overflow
        (np.nextafter(fmax + ulp / 2, 0.0), 0x7F7FFFFF),
        (2.0 ** -149, 0x00000001),
        (2.0 ** -150, 0x00000000),
        (np.nextafter(2.0 ** -150, 1.0), 0x00000001),
        (2.0 ** -126, 0x00800000),
        (1.0 + 2.0 ** -24, 0x3F800000),                     # tie -> even (1.0)
        (1.0 + 3 * 2.0 ** -24, 0x3F800002),                 # tie -> even (up)
    ]
    for x, want in cases:
        assert int(oracle.round_bits(np.array([x]), "f32")[0]) == want, x
    assert np.array_equal(oracle.decode(np.array([0x00000001, 0x7F7FFFFF], dtype=np.uint32), "f32"),
                          np.array([2.0 ** -149, fmax]))


def test_rounding_error_within_unit_roundoff():
    # Sec. 3.2: |fl(x) - x| <= u |x| in the normal range, u = 2^-p
    x = np.random.default_rng(7).uniform(-1000, 1000, 100_000)
    for fmt in ("f32", "f16"):
        r = oracle.rounded(x, fmt)
        assert np.all(np.abs(r - x) <= oracle.UNIT_ROUNDOFF[fmt] * np.abs(x))


def test_round_pack_zero_fills_padding():
    src = np.random.default_rng(3).standard_normal((5, 7))
    for fmt in ("f64", "f32", "f16"):
        out = oracle.round_pack(src, fmt, ld=16)
        assert out.shape == (5, 16)
        assert np.all(out[:, 7:] == 0)
        assert np.array_equal(oracle.decode(out[:, :7], fmt), oracle.rounded(src, fmt))
    assert oracle.packed_ld(1) == 16 and oracle.packed_ld(16) == 16 and oracle.packed_ld(17) == 32


# ---------------------------------------------------------------------------
# bfloat16 (Sec. 3.2 precision table: 8 significand bits, binary32's exponent
# range).  numpy has no bfloat16; its values are decoded here as the binary32
# numbers whose upper 16 bits are the pattern, and the library pin is torch's
# binary32 -> bfloat16 conversion on inputs that are binary32 numbers (so that
# no intermediate rounding is involved).
# ---------------------------------------------------------------------------

def bf16_values(bits):
    return (np.asarray(bits, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def test_bf16_direct_conversion_not_double_rounding():
    # 1 + 2^-8 + 2^-40 lies just above the midpoint between 1 and 1 + 2^-7:
    # direct rounding gives 1 + 2^-7; via binary32 the 2^-40 is lost first and
    # the tie then rounds to even (1.0)
    x = 1.0 + 2.0 ** -8 + 2.0 ** -40
    assert oracle.round_bits(np.array([x]), "bf16")[0] == 0x3F81
    assert oracle.round_bits(np.array([1.0 + 2.0 ** -8]), "bf16")[0] == 0x3F80


def test_exhaustive_bf16_values_roundtrip():
    allbits = np.arange(65536, dtype=np.uint16)
    vals = bf16_values(allbits)
    finite = np.isfinite(vals)
    assert np.array_equal(oracle.round_bits(vals[finite], "bf16"), allbits[finite])
    dec = oracle.decode(allbits, "bf16")
    assert np.array_equal(np.isnan(dec), np.isnan(vals))
    ok = ~np.isnan(vals)
    assert np.array_equal(dec[ok], vals[ok])


def test_bf16_midpoints_ties_to_even():
    pos = np.arange(0, 0x7F80, dtype=np.uint16)          # +0 .. max finite
    lo, hi = bf16_values(pos[:-1]), bf16_values(pos[1:])
    mid = (lo + hi) / 2.0                                 # exact in binary64
    even = np.where(pos[:-1] % 2 == 0, pos[:-1], pos[1:])
    assert np.array_equal(oracle.round_bits(mid, "bf16"), even)
    assert np.array_equal(oracle.round_bits(np.nextafter(mid, np.inf), "bf16"), pos[1:])
    assert np.array_equal(oracle.round_bits(np.nextafter(mid, -np.inf), "bf16"), pos[:-1])
    assert np.array_equal(oracle.round_bits(-mid, "bf16"), even | 0x8000)


def test_bf16_special_values_and_thresholds():
    bmax = (2.0 - 2.0 ** -7) * 2.0 ** 127
    cases = [
        (0.0, 0x0000), (-0.0, 0x8000), (np.inf, 0x7F80), (-np.inf, 0xFF80),
        (bmax, 0x7F7F),                                   # largest finite
        ((2.0 - 2.0 ** -8) * 2.0 ** 127, 0x7F80),         # overflow midpoint ties to even -> inf
        (np.nextafter((2.0 - 2.0 ** -8) * 2.0 ** 127, 0.0), 0x7F7F),
        (2.0 ** -133, 0x0001),                            # smallest subnormal
        (2.0 ** -134, 0x0000),                            # half of it: tie to even -> 0
        (np.nextafter(2.0 ** -134, 1.0), 0x0001),
        (3 * 2.0 ** -134, 0x0002),                        # tie between 1 and 2 quanta -> 2
        (2.0 ** -126, 0x0080),                            # smallest normal
        (5e-324, 0x0000), (1e300, 0x7F80), (-1e300, 0xFF80),
    ]
    for x, want in cases:
        assert int(oracle.round_bits(np.array([x]), "bf16")[0]) == want, x
    nan = oracle.round_bits(np.array([np.nan, -np.nan]), "bf16")
    assert np.all((nan & 0x7F80) == 0x7F80) and np.all((nan & 0x007F) != 0)


def test_bf16_matches_torch_on_binary32_inputs():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(5)
    x = (rng.standard_normal(300_000) * np.exp2(rng.uniform(-140, 120, 300_000))).astype(np.float32)
    x[:2000] = rng.standard_normal(2000).astype(np.float32)
    want = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.round_bits(x.astype(np.float64), "bf16"), want)


def test_bf16_rounding_error_within_unit_roundoff():
    x = np.random.default_rng(8).uniform(-1000, 1000, 100_000)
    r = oracle.rounded(x, "bf16")
    assert np.all(np.abs(r - x) <= oracle.UNIT_ROUNDOFF["bf16"] * np.abs(x))
    assert np.max(np.abs(r - x) / np.abs(x)) > 0.9 * oracle.UNIT_ROUNDOFF["bf16"]   # the bound is attained
