"""GPU rounding / packing (lrc_round_factors) and widening, bit-exact against
the oracle's IEEE round-to-nearest-even conversion."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import bits, packed, to_dev

pytestmark = pytest.mark.gpu


def gpu_round_flat(lrc, x: np.ndarray, fmt: str, dev):
    t = to_dev(x.reshape(1, -1), dev)
    out = lrc.round_matrix(t, fmt, ld=x.size)
    torch.cuda.synchronize()
    return bits(out, fmt).reshape(-1)


def test_exhaustive_binary16_midpoints(lrc, cuda):
    pos = np.arange(0, 0x7C00, dtype=np.uint16)
    lo = pos[:-1].view(np.float16).astype(np.float64)
    hi = pos[1:].view(np.float16).astype(np.float64)
    mid = (lo + hi) / 2.0
    x = np.concatenate([lo, mid, np.nextafter(mid, np.inf), np.nextafter(mid, -np.inf), -mid,
                        [65504.0, 65519.999, 65520.0, -65520.0, 1e300, 5e-324, -0.0, 0.0,
                         np.inf, -np.inf, 1.0 + 2.0 ** -11 + 2.0 ** -40]])
    got = gpu_round_flat(lrc, x, "f16", cuda)
    want = oracle.round_bits(x, "f16")
    assert np.array_equal(got, want)


def test_nan_stays_nan_with_sign(lrc, cuda):
    x = np.array([np.nan, -np.nan, 1.0, np.nan])
    for fmt in ("f16", "f32"):
        got = gpu_round_flat(lrc, x, fmt, cuda)
        dec = oracle.decode(got, fmt)
        assert np.isnan(dec[[0, 1, 3]]).all() and dec[2] == 1.0


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_random_wide_range_bit_exact(lrc, cuda, fmt):
    rng = np.random.default_rng(12)
    span = (-30, 20) if fmt == "f16" else (-160, 140)
    x = rng.standard_normal(1_000_003) * np.exp2(rng.uniform(*span, 1_000_003))
    assert np.array_equal(gpu_round_flat(lrc, x, fmt, cuda), oracle.round_bits(x, fmt))


@pytest.mark.parametrize("fmt", ["f64", "f32", "f16"])
@pytest.mark.parametrize("rows,cols,ld_src", [(1, 1, 1), (7, 33, 33), (5, 34, 40), (3, 129, 131), (64, 512, 512)])
def test_packing_and_padding(lrc, cuda, fmt, rows, cols, ld_src):
    src = W.gaussian((rows, ld_src), rows * 1000 + cols)
    t = to_dev(src, cuda)
    ld = lrc.lrc_packed_ld(cols)
    dst = torch.full((rows, ld), 7, dtype=lrc.storage_dtype(fmt), device=cuda)
    lrc.lrc_round_factors(t, rows, cols, ld_src, dst, ld, fmt)
    torch.cuda.synchronize()
    want = oracle.round_pack(src[:, :cols], fmt, ld=ld)
    assert np.array_equal(bits(dst, fmt), want.view(bits(dst, fmt).dtype))


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_widen_is_exact(lrc, cuda, fmt):
    src = W.gaussian((17, 45), 3)
    p = packed(lrc, src, fmt, cuda)
    w = lrc.widen_matrix(p, fmt, 45)
    torch.cuda.synchronize()
    got = w.cpu().numpy()
    assert np.array_equal(got[:, :45], oracle.rounded(src, fmt))
    assert np.all(got[:, 45:] == 0)


def test_large_factor_set_bit_exact(lrc, cuda):
    cfg = W.MATRIX_CONFIGS["large"]
    f = W.matrix_factors(cfg, "f16")
    for fmt in ("f32", "f16"):
        for a in (f.U, f.Vt):
            p = packed(lrc, a, fmt, cuda)
            torch.cuda.synchronize()
            got = bits(p, fmt)[:, :a.shape[1]]
            assert np.array_equal(got, oracle.round_bits(a, fmt))


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_widen_special_values_exact(lrc, cuda, fmt):
    """Widening is exact for every class of value: signed zeros, subnormals,
    the largest finite values, infinities, NaN, and random normal numbers."""
    dt = np.float32 if fmt == "f32" else np.float16
    fi = np.finfo(dt)
    rng = np.random.default_rng(11)
    specials = np.array([0.0, -0.0, fi.tiny, -fi.tiny, fi.smallest_subnormal, -fi.smallest_subnormal,
                         float(fi.max), -float(fi.max), np.inf, -np.inf, np.nan, 1.0, -2.5], dtype=np.float64)
    normals = rng.standard_normal(300) * np.exp2(rng.integers(-10, 10, 300))
    subnormals = rng.uniform(-1, 1, 200) * float(fi.tiny)
    vals = np.concatenate([specials, normals, subnormals]).astype(dt)
    rows, cols = 8, 73                       # 513 values + padding, ragged rows
    src = np.zeros(rows * cols, dtype=dt)
    src[:vals.size] = vals
    src = src.reshape(rows, cols)
    ld = lrc.lrc_packed_ld(cols)
    p = torch.zeros((rows, ld), dtype=lrc.storage_dtype(fmt), device=cuda)
    p[:, :cols] = torch.from_numpy(src).to(cuda)
    w = lrc.widen_matrix(p, fmt, cols)
    torch.cuda.synchronize()
    got = w.cpu().numpy()[:, :cols]
    want = src.astype(np.float64)
    nan = np.isnan(want)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan].view(np.uint64), want[~nan].view(np.uint64))
