"""GPU small-batch apply on the tensor cores (lrc_apply with at most 64
queries in binary16 or bfloat16; Sec. 4.4 Eq. gpu_matrix_apply) against the
oracle on the same rounded inputs.  The shapes cross the kernels' edges:
one to four 128-rank tiles, n from under one 64-wide k-block to the largest
the path takes (512 k-blocks, eight a chunk), chunk counts that leave the last
cluster of eight chunks partly empty, rows of U beyond the last 128-row tile,
and 16-, 32- and 64-query MMA widths."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, oracle_inputs, packed, rel_fro

pytestmark = pytest.mark.gpu

FMTS = ["f16", "f16_o16", "bf16"]


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
@pytest.mark.parametrize("m,n,k,b", [
    (129, 7, 3, 5),            # n under one k-block, rows past the first tile
    (1, 64, 16, 9),            # one row of U, one k-block
    (777, 1000, 127, 16),      # one rank tile, 16 chunks: two full clusters
    (1000, 4097, 129, 17),     # two rank tiles (the second holds one rank), 32-query width
    (3001, 8192, 272, 31),     # three rank tiles, the sweep workload's rank
    (256, 4096, 512, 32),      # four rank tiles, largest rank
    (300, 32768, 64, 24),      # largest n: eight k-blocks a chunk
    (513, 2000, 200, 6),       # 32 chunks of one k-block, a ragged last one
    (257, 300, 40, 1),         # one query
    (100, 1000, 100, 3),       # a few queries
    (300, 5000, 130, 33),      # 64-query width, two rank tiles
    (129, 1000, 33, 48),
    (700, 3000, 272, 64),      # largest batch of the path
])
def test_small_batch_tc_vs_oracle(lrc, cuda, fmt, m, n, k, b):
    f = W.random_factors(m, n, k, seed=m + 5 * n + k)
    X = W.gaussian((b, n), b + 21)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X, fmt)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    err = rel_fro(got, want)
    assert err <= TOL[fmt], (fmt, err)
    assert not np.isnan(got).any()


@pytest.mark.parametrize("fmt", ["f16", "f16_o16"])
@pytest.mark.parametrize("m,n,k,b", [(300, 3000, 200, 24), (130, 700, 33, 5), (200, 4097, 300, 32)])
def test_small_batch_tc_integer_exact(lrc, cuda, fmt, m, n, k, b):
    # small integers: the chunk, cluster and tile sums are exact in binary32,
    # W = X V diag(s) is an integer below 2048 (exact in binary16, lo = 0),
    # so the output is exact (binary16 output: rounded once)
    U = W.integer_valued((m, k), 31, -2, 2)
    s = W.integer_valued((k,), 32, 1, 2)
    Vt = W.integer_valued((k, n), 33, -1, 1)
    X = W.integer_valued((b, n), 34, -1, 1)
    inter = oracle.apply(np.eye(k), s, Vt, X)
    assert np.max(np.abs(inter)) < 2048
    got = run_apply(lrc, cuda, U, s, Vt, X, fmt)
    want = oracle.apply(U, s, Vt, X)
    if fmt == "f16_o16":
        want = oracle.rounded(want, "f16")
    assert np.array_equal(got, want), fmt


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("b", [2, 5, 16, 32, 64])
def test_small_batch_tc_bitwise_reproducible(lrc, cuda, fmt, b):
    m, n, k = 1500, 6000, 272
    f = W.random_factors(m, n, k, seed=b + 61)
    X = W.gaussian((b, n), b + 62)
    Ud, Sd, Vd, Xd = (packed(lrc, a, fmt, cuda) for a in (f.U, f.s, f.Vt, X))
    outs = []
    for _ in range(3):
        Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=cuda)
        lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, fmt)
        torch.empty(1 << 22, device=cuda).uniform_()       # unrelated work between the calls
        outs.append(Y.clone())
    assert lrc.lrc_device_status() == 0
    for y in outs[1:]:
        assert torch.equal(outs[0].view(torch.int16), y.view(torch.int16)) if y.element_size() == 2 else \
            torch.equal(outs[0].view(torch.int32), y.view(torch.int32))
    assert not torch.isnan(outs[0].double()).any()


def test_small_batch_tc_then_other_batches(lrc, cuda):
    """The arrival counters the path shares with the CUDA-core small-batch
    kernels are left at zero: calls of both kinds (rank 600 takes the CUDA
    cores), interleaved, match the oracle."""
    m, n, k = 900, 5000, 150
    g = W.random_factors(m, n, 600, seed=73)
    f = W.random_factors(m, n, k, seed=71)
    for b in (3, 20, 1, 64, 4, 9):
        X = W.gaussian((b, n), 72 + b)
        for h in ((f, g) if b <= 4 else (f,)):        # binary16 at rank 600: four queries at most
            got = run_apply(lrc, cuda, h.U, h.s, h.Vt, X, "f16")
            want = oracle.apply(*oracle_inputs(h.U, h.s, h.Vt, X, "f16"))
            assert rel_fro(got, want) <= TOL["f16"], (b, h.s.size)
