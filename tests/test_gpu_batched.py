"""Batched apply (lrc_apply_batched): several factor sets applied in one call,
the aggregate the paper times over a set of matrices (Sec. 4.4).  Each
problem is compared with the oracle on its own rounded inputs, and with the
single-problem lrc_apply; the tensor-core formats run every problem of a
group of 16 in one launch per phase."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, oracle_inputs, packed, rel_fro

pytestmark = pytest.mark.gpu

FMTS = ["f64", "f32", "f16", "f16_o16", "bf16", "f32tc"]


def problems(seed, count, mn=(300, 1138), k=41, b=(1, 600)):
    """Seeded problems of the paper's matrix sizes (m, n at most 1138)."""
    rng = np.random.default_rng(seed)
    out = []
    for p in range(count):
        m, n = (int(v) for v in rng.integers(mn[0], mn[1] + 1, size=2))
        bb = int(rng.integers(b[0], b[1] + 1))
        f = W.random_factors(m, n, k, seed=seed * 100 + p)
        X = W.gaussian((bb, n), seed * 100 + p + 50)
        out.append((f, X))
    return out


def run_batched(lrc, dev, probs, fmt):
    Us, Ss, Vs, Xs, Ys, ms, ns, ks, bs = ([] for _ in range(9))
    for f, X in probs:
        m, k = f.U.shape
        n = f.Vt.shape[1]
        b = X.shape[0]
        Us.append(packed(lrc, f.U, fmt, dev))
        Ss.append(packed(lrc, f.s, fmt, dev))
        Vs.append(packed(lrc, f.Vt, fmt, dev))
        Xs.append(packed(lrc, X, fmt, dev))
        Ys.append(torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=dev))
        ms.append(m), ns.append(n), ks.append(k), bs.append(b)
    lrc.lrc_apply_batched(Us, Ss, Vs, Xs, Ys, ms, ns, ks, bs, fmt)
    assert lrc.lrc_device_status() == 0
    return [y.double().cpu().numpy() for y in Ys], (Us, Ss, Vs, Xs)


def run_single(lrc, dev, ops, f, X, fmt):
    U, S, V, Xd = ops
    m, k = f.U.shape
    n, b = f.Vt.shape[1], X.shape[0]
    Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=dev)
    lrc.lrc_apply(U, S, V, Xd, Y, m, n, k, b, fmt)
    return Y.double().cpu().numpy()


@pytest.mark.parametrize("fmt", FMTS)
def test_batched_matches_oracle_and_single_calls(lrc, cuda, fmt):
    probs = problems(3, 10)
    got, ops = run_batched(lrc, cuda, probs, fmt)
    for p, ((f, X), y) in enumerate(zip(probs, got)):
        want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
        assert rel_fro(y, want) <= TOL[fmt], (fmt, p)
        single = run_single(lrc, cuda, tuple(o[p] for o in ops), f, X, fmt)
        assert rel_fro(y, single) <= 2 * TOL[fmt], (fmt, p)


@pytest.mark.parametrize("fmt", ["f16", "f16_o16", "bf16"])
def test_batched_mixed_shapes_and_more_than_one_group(lrc, cuda, fmt):
    """20 problems (two launch groups) with ragged sizes, rank 1 to 272,
    batches from 1 (many partials per entry: the sliced reduction) to 3000
    (the plain one) in the same group."""
    rng = np.random.default_rng(9)
    probs = []
    for p in range(20):
        m, n = (int(v) for v in rng.integers(17, 1500, size=2))
        k = int(rng.choice([1, 7, 41, 144, 272]))
        b = int(rng.choice([1, 3, 130, 3000]))
        f = W.random_factors(m, n, k, seed=700 + p)
        probs.append((f, W.gaussian((b, n), 800 + p)))
    got, _ = run_batched(lrc, cuda, probs, fmt)
    for p, ((f, X), y) in enumerate(zip(probs, got)):
        rows = W.sample_indices(min(X.shape[0], 48), X.shape[0], p)
        want = oracle.apply_rows(*oracle_inputs(f.U, f.s, f.Vt, X, fmt), rows)
        assert rel_fro(y[rows], want) <= TOL[fmt], (fmt, p, f.U.shape, X.shape)
        assert np.isfinite(y).all()


def test_batched_paper_scale_sampled(lrc, cuda):
    """Ten problems at the paper's batch (8192 queries), rank 41, binary16
    output; 64 sampled rows per problem."""
    probs = problems(11, 10, b=(8192, 8192))
    got, _ = run_batched(lrc, cuda, probs, "f16_o16")
    for p, ((f, X), y) in enumerate(zip(probs, got)):
        rows = W.sample_indices(64, X.shape[0], p + 1)
        want = oracle.apply_rows(*oracle_inputs(f.U, f.s, f.Vt, X, "f16_o16"), rows)
        assert rel_fro(y[rows], want) <= TOL["f16_o16"], p


def test_batched_bitwise_reproducible(lrc, cuda):
    probs = problems(5, 6)
    a, ops = run_batched(lrc, cuda, probs, "f16")
    b, _ = run_batched(lrc, cuda, probs, "f16")
    for x, y in zip(a, b):
        assert np.array_equal(x.view(np.uint64), y.view(np.uint64))


def test_batched_validation_names_the_problem(lrc, cuda):
    probs = problems(7, 3)
    Us = [packed(lrc, f.U, "f16", cuda) for f, _ in probs]
    Ss = [packed(lrc, f.s, "f16", cuda) for f, _ in probs]
    Vs = [packed(lrc, f.Vt, "f16", cuda) for f, _ in probs]
    Xs = [packed(lrc, X, "f16", cuda) for _, X in probs]
    Ys = [torch.full((X.shape[0], f.U.shape[0]), 7.0, device=cuda) for f, X in probs]
    ms = [f.U.shape[0] for f, _ in probs]
    ns = [f.Vt.shape[1] for f, _ in probs]
    ks = [f.U.shape[1] for f, _ in probs]
    bs = [X.shape[0] for _, X in probs]
    L = lrc.load()
    import ctypes
    arr = lambda ts: (ctypes.c_void_p * 3)(*[t.data_ptr() for t in ts])   # noqa: E731
    i64 = lambda xs: (ctypes.c_int64 * 3)(*xs)                            # noqa: E731
    bad_k = list(ks)
    bad_k[2] = 0
    st = L.lrc_apply_batched(3, arr(Us), arr(Ss), arr(Vs), arr(Xs), arr(Ys), i64(ms), i64(ns), i64(bad_k), i64(bs),
                             2, None)
    assert st == -1 and b"problem 2" in L.lrc_last_error()
    torch.cuda.synchronize()
    assert all(bool((y == 7.0).all()) for y in Ys)          # nothing was launched
    assert L.lrc_apply_batched(0, None, None, None, None, None, None, None, None, None, 2, None) == 0
