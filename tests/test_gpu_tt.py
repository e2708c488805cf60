"""GPU dense TT reconstruction (tt_reconstruct; Sec. 5.1 and Sec. 7.5
Eq. gpu_tt_reconstruction) against the oracle on the same rounded cores."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, base_fmt, rel_fro, to_dev

pytestmark = pytest.mark.gpu

FMTS = ["f64", "f32", "f16", "f16_o16", "f32tc"]


def run_tt(lrc, dev, cores64, fmt):
    b = base_fmt(fmt)
    rc = [oracle.rounded(c, b) for c in cores64]
    dc = [to_dev(c, dev).to(lrc.storage_dtype(fmt)).contiguous() for c in rc]
    dims = [c.shape[1] for c in cores64]
    ranks = [1] + [c.shape[2] for c in cores64]
    out = torch.full((int(np.prod(dims)),), float("nan"), dtype=lrc.output_dtype(fmt), device=dev)
    lrc.tt_reconstruct(dc, dims, ranks, fmt, out)
    torch.cuda.synchronize()
    return out.double().cpu().numpy(), rc


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", [
    ((3, 4), (1, 2, 1)),
    ((5, 7, 3), (1, 2, 3, 1)),
    ((2, 3, 2, 3, 2), (1, 2, 3, 3, 2, 1)),
    ((1, 9, 1, 4), (1, 1, 2, 2, 1)),
    ((300, 5), (1, 4, 1)),
])
def test_integer_cores_exact(lrc, cuda, fmt, dims, ranks):
    cores = [W.integer_valued((ranks[l], dims[l], ranks[l + 1]), 50 + l, -2, 2) for l in range(len(dims))]
    got, rc = run_tt(lrc, cuda, cores, fmt)
    want = oracle.tt_full(rc).reshape(-1)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,r,kind", [
    ((37, 29, 41), 9, "gauss_geo"),
    ((8, 9, 7, 6, 5), 11, "gauss_alg"),
    ((130, 70), 33, "gauss_geo"),
    ((64, 48, 224), 52, "smooth"),
    ((16,) * 5, 28, "gauss_alg"),
])
def test_random_cores_vs_oracle(lrc, cuda, fmt, dims, r, kind):
    cores = W.make_tt(dims, W.capped_ranks(dims, r), kind, 17)
    got, rc = run_tt(lrc, cuda, cores, fmt)
    want = oracle.tt_full(rc).reshape(-1)
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)


# narrow last two modes (the binary16 path batches all i_{d-1} in one product):
# d = 3, 4, 5; ragged prefix count; rank padding in both products; a
# non-square last pair
NARROW = [
    ((3, 16, 16), (1, 3, 16, 1)),
    ((4, 5, 16, 16), (1, 3, 7, 16, 1)),
    ((2, 3, 4, 16, 16), (1, 2, 6, 20, 16, 1)),
    ((5, 8, 32), (1, 4, 8, 1)),
    ((257, 16, 16), (1, 9, 12, 1)),
    ((70, 4, 64), (1, 33, 16, 1)),
]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", NARROW)
def test_narrow_last_modes_vs_oracle(lrc, cuda, fmt, dims, ranks):
    cores = W.make_tt(dims, ranks, "gauss_geo", 23)
    got, rc = run_tt(lrc, cuda, cores, fmt)
    want = oracle.tt_full(rc).reshape(-1)
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)


@pytest.mark.parametrize("fmt", ["f16"])
@pytest.mark.parametrize("dims,ranks", NARROW)
def test_narrow_last_modes_integer_exact(lrc, cuda, fmt, dims, ranks):
    # small integers: every product and partial sum is exact, and the hi/lo
    # split represents every intermediate exactly
    cores = [W.integer_valued((ranks[l], dims[l], ranks[l + 1]), 70 + l, -1, 1) for l in range(len(dims))]
    got, rc = run_tt(lrc, cuda, cores, fmt)
    want = oracle.tt_full(rc).reshape(-1)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("name", ["tt3", "tt6", "tt_hsi"])
def test_workloads_sampled_entries(lrc, cuda, fmt, name):
    """The three TT workloads at full size, in the bench's launch
    configuration; 20000 seeded entries checked with the oracle's
    independent entry evaluator."""
    cfg = W.TT_CONFIGS[name]
    cores = W.tt_cores(cfg, base_fmt(fmt))
    got, rc = run_tt(lrc, cuda, cores, fmt)
    idx = W.sample_indices(20000, got.size, 3)
    want = oracle.tt_entries(rc, idx)
    err = rel_fro(got[idx], want)
    assert err <= TOL[fmt], (name, fmt, err)
    assert np.isfinite(got).all()


# Interior cores too large for the small-core product-chain path's shared
# memory: these shapes take the narrow-mode tensor-core kernel (last two
# modes 16 x 16) and the d >= 4 wide-mode kernel (last mode 64).
LARGE_CORES = [
    ((8, 128, 16, 16), (1, 8, 64, 16, 1)),
    ((8, 128, 8, 64), (1, 8, 64, 32, 1)),
]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", LARGE_CORES)
def test_large_interior_cores_vs_oracle(lrc, cuda, fmt, dims, ranks):
    cores = W.make_tt(dims, ranks, "gauss_geo", 31)
    got, rc = run_tt(lrc, cuda, cores, fmt)
    want = oracle.tt_full(rc).reshape(-1)
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)
    assert np.isfinite(got).all()


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", [
    ((64, 48, 80), (1, 12, 9, 1)),           # 3-way, wide last mode
    ((8, 8, 8, 8, 8), (1, 6, 7, 7, 6, 1)),   # narrow modes, chain meeting in the middle
])
def test_tt_bitwise_reproducible(lrc, cuda, fmt, dims, ranks):
    """Two reconstructions of the same cores agree bit for bit."""
    cores = [W.gaussian((ranks[l], dims[l], ranks[l + 1]), 90 + l) for l in range(len(dims))]
    a, _ = run_tt(lrc, cuda, cores, fmt)
    torch.empty(1 << 22, device=cuda).uniform_()
    b, _ = run_tt(lrc, cuda, cores, fmt)
    assert np.array_equal(a.view(np.uint64), b.view(np.uint64)), fmt
    assert np.isfinite(a).all()
