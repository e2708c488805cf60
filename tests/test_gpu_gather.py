"""Sampled TT entries (tt_gather; Sec. 5.1, T(i_1..i_d) = G_1(i_1)...G_d(i_d))
against the oracle's independent entry evaluator on the same rounded cores."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, base_fmt, rel_fro, to_dev

pytestmark = pytest.mark.gpu

FMTS = ["f64", "f32", "f16", "f16_o16"]


def gather(lrc, dev, cores, fmt, idx):
    dims = [c.shape[1] for c in cores]
    ranks = [1] + [c.shape[2] for c in cores]
    rounded = [oracle.rounded(c, base_fmt(fmt)) for c in cores]
    dc = [to_dev(c, dev).to(lrc.storage_dtype(fmt)).contiguous() for c in rounded]
    di = to_dev(np.ascontiguousarray(idx, dtype=np.int64), dev)
    out = torch.empty(len(idx), dtype=lrc.output_dtype(fmt), device=dev)
    lrc.tt_gather(dc, dims, ranks, fmt, di, out)
    torch.cuda.synchronize()
    return out.double().cpu().numpy(), rounded


SHAPES = [
    ((37, 29), (1, 5, 1)),
    ((7, 9, 11), (1, 3, 4, 1)),
    ((5, 6, 7, 8), (1, 4, 9, 6, 1)),
    ((4,) * 6, (1, 4, 8, 8, 8, 4, 1)),
    ((300, 2, 40), (1, 33, 17, 1)),
    ((3, 16, 16), (1, 3, 16, 1)),
    ((300, 250), (1, 200, 1)),
    ((120, 90, 80), (1, 100, 70, 1)),
]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", SHAPES)
def test_gather_vs_oracle(lrc, cuda, fmt, dims, ranks):
    cores = W.make_tt(dims, ranks, "gauss_geo", 31 + sum(dims))
    total = int(np.prod(dims))
    idx = W.sample_indices(min(total, 5000), total, 3)
    got, rounded = gather(lrc, cuda, cores, fmt, idx)
    want = oracle.tt_entries(rounded, idx)
    assert rel_fro(got, want) <= TOL[fmt], rel_fro(got, want)


@pytest.mark.parametrize("fmt", ["f64", "f32", "f16", "f16_o16"])
def test_gather_integer_cores_exact(lrc, cuda, fmt):
    """Small-integer cores: every product and sum is exact in every format."""
    dims, ranks = (6, 5, 7, 4), (1, 3, 4, 2, 1)
    cores = [W.integer_valued((ranks[l], dims[l], ranks[l + 1]), 50 + l, -3, 3) for l in range(4)]
    idx = np.arange(int(np.prod(dims)), dtype=np.int64)
    got, rounded = gather(lrc, cuda, cores, fmt, idx)
    assert np.array_equal(got, oracle.tt_entries(rounded, idx))


@pytest.mark.parametrize("name", ["tt3", "tt6", "tt_hsi"])
@pytest.mark.parametrize("fmt", FMTS)
def test_gather_full_workloads(lrc, cuda, name, fmt):
    """The three TT workloads at their ranks of `fmt`, 20000 random (unsorted,
    repeated) indices."""
    cfg = W.TT_CONFIGS[name]
    cores = W.tt_cores(cfg, base_fmt(fmt))
    total = int(np.prod(cfg.dims))
    idx = np.random.default_rng(5).integers(0, total, size=20000).astype(np.int64)
    got, rounded = gather(lrc, cuda, cores, fmt, idx)
    want = oracle.tt_entries(rounded, idx)
    assert rel_fro(got, want) <= TOL[fmt], rel_fro(got, want)


def test_gather_out_of_range_and_empty(lrc, cuda):
    dims, ranks = (4, 5, 6), (1, 2, 3, 1)
    cores = W.make_tt(dims, ranks, "gauss", 3)
    total = int(np.prod(dims))
    idx = np.array([0, -1, total - 1, total, 7, 1 << 40], dtype=np.int64)
    got, rounded = gather(lrc, cuda, cores, "f64", idx)
    ok = np.array([True, False, True, False, True, False])
    assert np.all(np.isnan(got[~ok]))
    assert np.array_equal(got[ok], oracle.tt_entries(rounded, idx[ok]))
    # count 0: nothing launched, nothing written
    dc = [to_dev(c, cuda) for c in cores]
    before = lrc.lrc_launch_count()
    lrc.tt_gather(dc, dims, ranks, "f64", torch.empty(0, dtype=torch.int64, device=cuda),
                  torch.empty(0, dtype=torch.float64, device=cuda))
    assert lrc.lrc_launch_count() == before
