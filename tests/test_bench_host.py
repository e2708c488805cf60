"""Host logic of bench.py that every reported fraction rests on: the
algorithmic bytes and flops of each call (the roofline formulas for the apply,
the TT reconstruction, rounding and the Frobenius difference) and the
cheapest contraction of a TT chain -- checked without a GPU."""
import itertools

import numpy as np
import pytest

import bench


def mb(x):
    return x / 1e6


@pytest.mark.parametrize("fmt,k,want_mb,want_gflop", [
    ("f64", 128, 1636, 51.5),       # cfg 2, FP64 baseline
    ("f32", 136, 819, 54.8),        # cfg 2, FP32 at k' = 136
    ("f16", 144, 678, 58.0),        # cfg 2, FP16 with FP32 output
    ("f16_o16", 144, 410, 58.0),    # cfg 2, FP16 output
])
def test_apply_work_matches_the_table(fmt, k, want_mb, want_gflop):
    w = bench.work_apply(16384, 8192, k, 8192, fmt)
    assert mb(w["bytes"]) == pytest.approx(want_mb, rel=2e-3)
    assert w["flops"] / 1e9 == pytest.approx(want_gflop, rel=2e-3)


@pytest.mark.parametrize("b,fmt,want_mb", [
    (1, "f64", 67.4), (1, "f32", 35.8), (1, "f16", 17.9),
    (256, "f16", 43.0), (256, "f16_o16", 34.6),
    (4096, "f32", 573), (32768, "f16_o16", 2165),
])
def test_sweep_work_matches_the_table(b, fmt, want_mb):
    k = 256 if fmt == "f64" else 272
    assert mb(bench.work_apply(16384, 16384, k, b, fmt)["bytes"]) == pytest.approx(want_mb, rel=5e-3)


def brute_chain_flops(dims, ranks):
    """Cheapest product chain by enumeration: every bond c, the left side
    contracted left to right and the right side right to left, counted as
    2 x (rows x inner x cols) of each explicit matrix product."""
    d = len(dims)
    best = None
    for c in range(1, d):
        f = 0
        Z = (dims[0], ranks[1])                       # rows, cols of Z(1)
        for j in range(1, c):
            K = (ranks[j], dims[j] * ranks[j + 1])
            f += 2 * Z[0] * Z[1] * K[1]
            Z = (Z[0] * dims[j], ranks[j + 1])
        S = (ranks[d - 1], dims[d - 1])
        for j in range(d - 2, c - 1, -1):
            K = (ranks[j] * dims[j], ranks[j + 1])
            f += 2 * K[0] * K[1] * S[1]
            S = (ranks[j], dims[j] * S[1])
        assert Z[1] == S[0] == ranks[c]
        f += 2 * Z[0] * Z[1] * S[1]
        best = f if best is None else min(best, f)
    return best


@pytest.mark.parametrize("dims,ranks", [
    ((256, 256, 256), (1, 34, 34, 1)),
    ((16,) * 6, (1, 16, 26, 26, 26, 16, 1)),
    ((512, 512, 224), (1, 70, 52, 1)),
    ((3, 4), (1, 2, 1)),
    ((5, 7, 3, 2), (1, 2, 5, 3, 1)),
])
def test_tt_chain_flops_is_the_cheapest_chain(dims, ranks):
    assert bench.tt_chain_flops(dims, ranks) == brute_chain_flops(dims, ranks)


def test_tt_chain_flops_16pow6_saves_on_left_to_right():
    dims, ranks = (16,) * 6, (1, 16, 26, 26, 26, 16, 1)
    ltr = sum(2 * int(np.prod(dims[:l])) * ranks[l] * dims[l] * ranks[l + 1] for l in range(1, 6))
    assert ltr / 1e9 == pytest.approx(1.50, rel=5e-3)         # the table's left-to-right count
    assert bench.tt_chain_flops(dims, ranks) <= 0.62 * ltr


def test_tt_work_matches_the_table():
    w = bench.work_tt((256, 256, 256), (1, 34, 34, 1), "f16")
    assert mb(w["bytes"]) == pytest.approx(67.7, rel=5e-3)
    w = bench.work_tt((256, 256, 256), (1, 34, 34, 1), "f16_o16")
    assert mb(w["bytes"]) == pytest.approx(34.2, rel=5e-3)


def test_roofline_takes_the_larger_bound():
    w = bench.work_apply(16384, 8192, 144, 8192, "f16")
    t_hbm = w["bytes"] / bench.PEAKS["hbm"]
    assert bench.roofline_time(w) == pytest.approx(max(t_hbm, w["flops"] / bench.PEAKS["f16"]))
    assert bench.bound_of(w) == "hbm"
    w64 = bench.work_apply(16384, 8192, 128, 8192, "f64")
    assert bench.bound_of(w64) == "alu"


def test_f32tc_bound_adds_the_two_engines():
    m, n, k, b = 16384, 8192, 136, 8192
    w = bench.work_apply(m, n, k, b, "f32tc")
    want = 2 * n * k * b / bench.PEAKS["f32"] + 3 * 2 * m * k * b / bench.PEAKS["f16"]
    assert w["alu_time"] == pytest.approx(want)
    assert bench.roofline_time(w) == pytest.approx(max(w["bytes"] / bench.PEAKS["hbm"], want))
    assert w["bytes"] == bench.work_apply(m, n, k, b, "f32")["bytes"]
