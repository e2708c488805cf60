"""GPU batched low-rank apply (lrc_apply, Sec. 4.4 Eq. gpu_matrix_apply)
against the oracle evaluated on the same rounded inputs."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, base_fmt, oracle_inputs, packed, rel_fro

pytestmark = pytest.mark.gpu

FMTS = ["f64", "f32", "f16", "f16_o16", "f32tc"]


def run_apply(lrc, dev, U, s, Vt, X, fmt):
    m, k = U.shape
    n = Vt.shape[1]
    b = X.shape[0]
    Ud, Sd, Vd, Xd = (packed(lrc, a, fmt, dev) for a in (U, s, Vt, X))
    Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=dev)
    lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, fmt)
    assert lrc.lrc_device_status() == 0
    return Y.double().cpu().numpy()


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("m,n,k,b", [(40, 24, 5, 3), (130, 70, 33, 17), (257, 129, 144, 129)])
def test_integer_inputs_exact(lrc, cuda, fmt, m, n, k, b):
    # small integers: every product and partial sum is exact in every format
    U = W.integer_valued((m, k), 1, -2, 2)
    s = W.integer_valued((k,), 2, 1, 2)
    Vt = W.integer_valued((k, n), 3, -2, 2)
    X = W.integer_valued((b, n), 4, -2, 2)
    got = run_apply(lrc, cuda, U, s, Vt, X, fmt)
    want = oracle.apply(U, s, Vt, X)
    if fmt == "f16_o16":
        # the binary16 intermediate X V diag(s) stays an exact integer (< 2048),
        # every FP32 partial sum is exact, and the output is rounded once
        assert np.max(np.abs(oracle.apply(np.eye(k), s, Vt, X))) < 2048
        want = oracle.rounded(want, "f16")
    assert np.array_equal(got, want), fmt


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("m,n,k,b", [
    (512, 512, 34, 64),        # tiny workload shape
    (100, 300, 1, 1),          # rank 1, single query
    (1000, 136, 136, 7),       # k = n
    (48, 40, 60, 5),           # k > min(m, n)
    (777, 1029, 272, 250),     # ragged everything, rank of the sweep workload
    (2048, 1536, 144, 300),
])
def test_random_factors_vs_oracle(lrc, cuda, fmt, m, n, k, b):
    f = W.random_factors(m, n, k, seed=m + n + k)
    X = W.gaussian((b, n), b + 5)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)


@pytest.mark.parametrize("fmt", FMTS)
def test_tiny_workload_full(lrc, cuda, fmt):
    cfg = W.MATRIX_CONFIGS["tiny"]
    f = W.matrix_factors(cfg, base_fmt(fmt))
    X = W.queries(cfg)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    assert rel_fro(got, want) <= TOL[fmt]


@pytest.mark.parametrize("fmt", FMTS)
def test_large_workload_sampled_rows(lrc, cuda, fmt):
    """m = 16384, n = 8192, b = 8192 in the bench's launch configuration;
    256 seeded query rows are checked against the oracle."""
    cfg = W.MATRIX_CONFIGS["large"]
    f = W.matrix_factors(cfg, base_fmt(fmt))
    X = W.queries(cfg)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    rows = W.sample_indices(256, cfg.b, 99)
    Ur, sr, Vr, Xr = oracle_inputs(f.U, f.s, f.Vt, X, fmt)
    want = oracle.apply_rows(Ur, sr, Vr, Xr, rows)
    err = rel_fro(got[rows], want)
    assert err <= TOL[fmt], (fmt, err)
    assert np.isfinite(got).all()


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("b", [1, 16, 256])
def test_sweep_workload_small_batches(lrc, cuda, fmt, b):
    cfg = W.sweep_config(b)
    f = W.matrix_factors(cfg, base_fmt(fmt))
    X = W.queries(cfg)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    rows = W.sample_indices(min(b, 32), b, 7)
    want = oracle.apply_rows(*oracle_inputs(f.U, f.s, f.Vt, X, fmt), rows)
    assert rel_fro(got[rows], want) <= TOL[fmt]


def test_identity_queries_reconstruct_dense_f64(lrc, cuda):
    # X = I_n gives A_k^T: the dense FP64 reconstruction used for eta
    f = W.random_factors(300, 200, 20, seed=3)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, np.eye(200), "f64")
    want = (f.Vt.T * f.s) @ f.U.T
    assert np.max(np.abs(got - want)) <= 1e-14 * np.max(np.abs(want))


@pytest.mark.parametrize("fmt", ["f32", "f64", "f32tc"])
@pytest.mark.parametrize("m,n,k,b", [
    (257, 1100, 136, 300),     # several n-splits, one 160-wide rank tile
    (130, 3000, 161, 517),     # rank above 160: two rank tiles, ragged everything
    (40, 24, 5, 2100),         # n shorter than one slab
])
def test_large_batch_integer_exact(lrc, cuda, fmt, m, n, k, b):
    # batches above the small-batch split path: every product and partial sum
    # of the register-tiled products is an exact integer below 2^24
    U = W.integer_valued((m, k), 11, -2, 2)
    s = W.integer_valued((k,), 12, 1, 2)
    Vt = W.integer_valued((k, n), 13, -2, 2)
    X = W.integer_valued((b, n), 14, -2, 2)
    got = run_apply(lrc, cuda, U, s, Vt, X, fmt)
    assert np.array_equal(got, oracle.apply(U, s, Vt, X)), fmt


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("m,n,k,b", [
    (333, 1031, 37, 5),        # ragged n (not a whole number of 16-byte vectors), b between the kernel's widths
    (64, 7, 3, 16),            # n shorter than one vector row, largest batch of the small-batch kernels
    (1000, 5000, 272, 16),     # several n-chunks with a ragged last chunk
    (4097, 2049, 1024, 2),     # largest rank of the small-batch kernels
    (517, 3001, 100, 4),       # largest batch of the small-batch kernels for FP16
    (600, 2500, 200, 12),      # 16-query kernels (two rows of V^T per warp for FP64)
    (301, 777, 45, 8),         # 8-query kernels
    (257, 129, 19, 1),         # single query, ragged everything
])
def test_small_batch_kernels_vs_oracle(lrc, cuda, fmt, m, n, k, b):
    f = W.random_factors(m, n, k, seed=m + 3 * n + k)
    X = W.gaussian((b, n), b + 11)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("b", [1, 4, 16, 200, 3000])
def test_apply_bitwise_reproducible(lrc, cuda, fmt, b):
    """Every batch regime (small-batch streams, split products, the
    tensor-core path with its sliced partial reduction, stream-K partials)
    adds in a fixed order: two calls on the same inputs agree bit for bit,
    with other work queued on the stream in between."""
    m, n, k = 700, 2100, 72
    f = W.random_factors(m, n, k, seed=b + 41)
    X = W.gaussian((b, n), b + 42)
    Ud, Sd, Vd, Xd = (packed(lrc, a, fmt, cuda) for a in (f.U, f.s, f.Vt, X))
    outs = []
    for _ in range(2):
        Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=cuda)
        lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, fmt)
        torch.empty(1 << 22, device=cuda).uniform_()       # unrelated work between the calls
        outs.append(Y.clone())
    assert lrc.lrc_device_status() == 0
    assert torch.equal(outs[0].view(torch.int8), outs[1].view(torch.int8)), (fmt, b)
    assert not torch.isnan(outs[0].double()).any()


@pytest.mark.parametrize("m,n,k,b", [
    (2048, 1536, 136, 300),    # rank of the large-batch workload, ragged batch: the tensor-core product
    (1000, 700, 192, 129),     # largest rank of the tensor-core product
    (900, 600, 200, 64),       # rank above it: the binary32 product kernel
])
def test_f32tc_matches_f32_path(lrc, cuda, m, n, k, b):
    """LRC_F32_TC (second product on the tensor cores through the scaled
    binary16 hi/lo split) stays within the binary32 tolerance of the oracle
    and of the LRC_F32 result on the same inputs."""
    f = W.random_factors(m, n, k, seed=m + k + 7)
    X = W.gaussian((b, n), b + 3)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, "f32"))
    got_tc = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, "f32tc")
    got_32 = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, "f32")
    assert rel_fro(got_tc, want) <= TOL["f32tc"]
    assert rel_fro(got_tc, got_32) <= 2 * TOL["f32"]


def test_f32tc_wide_dynamic_range(lrc, cuda):
    """Queries spanning 40 binades and factor rows spanning 16: W takes a
    power-of-two scale per row and U one per 32 rows, so every part stays a
    normal binary16 number and each query keeps binary32 accuracy."""
    m, n, k, b = 512, 384, 96, 256
    f = W.random_factors(m, n, k, seed=77)
    rng = np.random.default_rng(78)
    U = f.U * np.exp2(rng.integers(-8, 8, size=(m, 1)))
    X = W.gaussian((b, n), 79) * np.exp2(rng.integers(-20, 20, size=(b, 1)))
    want = oracle.apply(*oracle_inputs(U, f.s, f.Vt, X, "f32"))
    got = run_apply(lrc, cuda, U, f.s, f.Vt, X, "f32tc")
    # per-row relative error: every query row is judged against its own scale
    err = np.linalg.norm(got - want, axis=1) / np.linalg.norm(want, axis=1)
    assert err.max() <= 1e-5, err.max()


@pytest.mark.parametrize("fmt", ["f16_o16", "bf16"])
@pytest.mark.parametrize("m,n,k,b", [
    (2000, 3000, 100, 777),    # two k-blocks, ragged m and b: U resident, W streamed
    (5000, 2000, 160, 1300),   # three k-blocks; CTAs whose ranges cross column tiles
    (300, 700, 129, 2000),     # a single column tile, many row tiles
])
def test_resident_u_product_vs_oracle(lrc, cuda, fmt, m, n, k, b):
    """16-bit-output applies whose second product keeps U resident per
    column tile (several k-blocks, one plane of W) match the oracle and are
    reproducible bit for bit."""
    f = W.random_factors(m, n, k, seed=m + 7 * k)
    X = W.gaussian((b, n), b + 91)
    Ud, Sd, Vd, Xd = (packed(lrc, a, fmt, cuda) for a in (f.U, f.s, f.Vt, X))
    outs = []
    for _ in range(2):
        Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=cuda)
        lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, fmt)
        outs.append(Y)
    assert lrc.lrc_device_status() == 0
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    err = rel_fro(outs[0].double().cpu().numpy(), want)
    assert err <= TOL[fmt], (fmt, err)
