"""Pins for the oracle's TT reconstruction: the chain of Sec. 7.5
(Eq. gpu_tt_reconstruction) and the entry evaluator of Sec. 5.1.

Independent facts used: brute-force sums over every rank-index path (pure
Python), tensors of known TT rank with closed-form entries, invariance under
zero rank padding and under a gauge change M M^-1 (Sec. 6.1), and the norm
identity ||T||_F = ||lambda||_2 of the left-orthogonal generator.
"""
import itertools
import math

import numpy as np
import pytest

import oracle
import workloads as W


def brute_tt(cores):
    """T(i) = sum over rank paths a_1..a_{d-1} of prod_l G_l[a_{l-1}, i_l, a_l]."""
    dims = [c.shape[1] for c in cores]
    ranks = [1] + [c.shape[2] for c in cores]
    out = np.zeros(dims)
    for idx in itertools.product(*[range(n) for n in dims]):
        total = 0.0
        for path in itertools.product(*[range(r) for r in ranks[1:-1]]):
            a = (0,) + path + (0,)
            prod = 1.0
            for l, c in enumerate(cores):
                prod *= c[a[l], idx[l], a[l + 1]]
            total += prod
        out[idx] = total
    return out


@pytest.mark.parametrize("dims,ranks", [
    ((3, 4), (1, 2, 1)),
    ((3, 4, 2), (1, 2, 3, 1)),
    ((2, 3, 2, 3), (1, 2, 3, 2, 1)),
    ((5, 1, 4), (1, 1, 3, 1)),
])
def test_chain_and_entries_equal_brute_force_on_integers(dims, ranks):
    cores = [W.integer_valued((ranks[l], dims[l], ranks[l + 1]), 100 + l, -3, 3)
             for l in range(len(dims))]
    want = brute_tt(cores)
    got = oracle.tt_full(cores)
    assert got.shape == tuple(dims)
    assert np.array_equal(got, want)
    flat = np.arange(want.size)
    assert np.array_equal(oracle.tt_entries(cores, flat), want.reshape(-1))


def test_chain_entries_agree_on_gaussian_cores():
    dims, ranks = (6, 5, 7, 4), (1, 3, 4, 2, 1)
    cores = W.make_tt(dims, ranks, "gauss", 77)
    full = oracle.tt_full(cores)
    idx = W.sample_indices(300, full.size, 5)
    ent = oracle.tt_entries(cores, idx)
    assert np.max(np.abs(ent - full.reshape(-1)[idx])) <= 1e-14 * np.max(np.abs(full))


def test_sum_of_univariate_functions_rank2():
    # T(i) = sum_l f_l(i_l): cores [f_1 1], [[1 0],[f_l 1]], [1; f_d]
    dims = (4, 3, 5, 2)
    rng = np.random.default_rng(3)
    fs = [rng.standard_normal(n) for n in dims]
    d = len(dims)
    cores = []
    for l, n in enumerate(dims):
        if l == 0:
            c = np.zeros((1, n, 2)); c[0, :, 0] = fs[0]; c[0, :, 1] = 1.0
        elif l == d - 1:
            c = np.zeros((2, n, 1)); c[0, :, 0] = 1.0; c[1, :, 0] = fs[l]
        else:
            c = np.zeros((2, n, 2)); c[0, :, 0] = 1.0; c[1, :, 0] = fs[l]; c[1, :, 1] = 1.0
        cores.append(c)
    want = sum(np.reshape(fs[l], [dims[l] if q == l else 1 for q in range(d)]) for l in range(d))
    assert np.allclose(oracle.tt_full(cores), want, rtol=0, atol=1e-14)


def test_sine_of_sum_rank2():
    # sin(x_1 + ... + x_d) by the angle-addition cores
    dims = (7, 6, 5)
    xs = [np.linspace(0.1, 2.0, n) * (l + 1) for l, n in enumerate(dims)]
    c1 = np.stack([np.sin(xs[0]), np.cos(xs[0])], axis=-1)[None]          # 1 x n x 2
    c2 = np.zeros((2, dims[1], 2))
    c2[0, :, 0] = np.cos(xs[1]); c2[0, :, 1] = -np.sin(xs[1])
    c2[1, :, 0] = np.sin(xs[1]); c2[1, :, 1] = np.cos(xs[1])
    c3 = np.zeros((2, dims[2], 1))
    c3[0, :, 0] = np.cos(xs[2]); c3[1, :, 0] = np.sin(xs[2])
    want = np.sin(xs[0][:, None, None] + xs[1][None, :, None] + xs[2][None, None, :])
    got = oracle.tt_full([c1, c2, c3])
    assert np.max(np.abs(got - want)) <= 1e-15 * 8


def test_product_rank1():
    dims = (3, 8, 4, 5)
    fs = [np.random.default_rng(l).standard_normal(n) for l, n in enumerate(dims)]
    cores = [f.reshape(1, -1, 1) for f in fs]
    want = np.einsum("i,j,k,l->ijkl", *fs)
    assert np.allclose(oracle.tt_full(cores), want, rtol=1e-15, atol=0)


def test_zero_rank_padding_invariance():
    dims, ranks = (4, 5, 3), (1, 2, 3, 1)
    cores = W.make_tt(dims, ranks, "gauss", 9)
    padded = []
    pr = (1, 4, 6, 1)
    for l, c in enumerate(cores):
        p = np.zeros((pr[l], dims[l], pr[l + 1]))
        p[:c.shape[0], :, :c.shape[2]] = c
        padded.append(p)
    assert np.array_equal(oracle.tt_full(padded), oracle.tt_full(cores))


def test_gauge_invariance():
    # inserting M M^-1 between cores 1 and 2 leaves T unchanged (Sec. 6.1)
    dims, ranks = (5, 4, 6), (1, 3, 3, 1)
    cores = W.make_tt(dims, ranks, "gauss", 21)
    M = np.random.default_rng(2).standard_normal((3, 3)) + 3 * np.eye(3)
    g1 = np.einsum("aib,bc->aic", cores[0], M)
    g2 = np.einsum("ab,bic->aic", np.linalg.inv(M), cores[1])
    T0 = oracle.tt_full(cores)
    T1 = oracle.tt_full([g1, g2, cores[2]])
    assert np.max(np.abs(T1 - T0)) <= 1e-13 * np.max(np.abs(T0))


@pytest.mark.parametrize("dims,r,kind", [((16, 12, 10), 5, "gauss_geo"), ((6,) * 4, 7, "gauss_alg")])
def test_left_orthogonal_generator_norm_identity(dims, r, kind):
    ranks = W.capped_ranks(dims, r)
    cores = W.make_tt(dims, ranks, kind, 31)
    lam = W.tt_last_spectrum(kind, ranks[-2])
    T = oracle.tt_full(cores)
    nrm, _ = oracle.fro_diff(T)
    assert abs(nrm - math.sqrt(float(np.sum(lam ** 2)))) <= 1e-13


def test_eta_tt_scale():
    # eta_TT of rounded left-orthogonal cores is of order u ||T|| (Sec. 6.1)
    dims = (20, 18, 16)
    cores = W.make_tt(dims, W.capped_ranks(dims, 6), "gauss_geo", 41)
    nrm, _ = oracle.fro_diff(oracle.tt_full(cores))
    for fmt in ("f32", "f16"):
        rel = oracle.eta_tt(cores, fmt) / nrm
        assert 0.2 * oracle.UNIT_ROUNDOFF[fmt] < rel < 2.0 * oracle.UNIT_ROUNDOFF[fmt]
