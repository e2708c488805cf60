"""Pins of the oracle's eta (Thm 4.1) and eta_TT (Thm 6.1) against exact
rational arithmetic on tiny inputs, and exact checks of the two identities
the fused eta kernels rest on:

  A - Ah = [dU, Uh] [[S, S], [S, dS]] [dV, Vh]^T       (dU = U - Uh, ...)
  [D_l, Zh_l] = [D_{l-1}, Zh_{l-1}] [[G_l, 0], [dG_l, Gh_l]],
  T - Th = [D_{d-1}, Zh_{d-1}] [G_d; dG_d]              (D_l = Z_l - Zh_l)

Rounding here is numpy's binary32 / binary16 conversion, independent of the
oracle's own rounding code."""
from fractions import Fraction
import itertools
import math

import numpy as np
import pytest

import oracle
import workloads as W

NP_DT = {"f32": np.float32, "f16": np.float16}


def rnd(a, fmt):
    return np.asarray(a, dtype=np.float64).astype(NP_DT[fmt]).astype(np.float64)


def F(a):
    return np.vectorize(Fraction, otypes=[object])(np.asarray(a, dtype=np.float64))


def exact_lowrank(U, s, Vt):
    m, k = U.shape
    n = Vt.shape[1]
    Uf, sf, Vf = F(U), F(s), F(Vt)
    return [[sum(Uf[i, l] * sf[l] * Vf[l, j] for l in range(k)) for j in range(n)] for i in range(m)]


def exact_tt(cores):
    dims = [c.shape[1] for c in cores]
    Cf = [F(c) for c in cores]
    out = {}
    for idx in itertools.product(*[range(x) for x in dims]):
        v = np.array([[Fraction(1)]], dtype=object)
        for c, i in zip(Cf, idx):
            v = v.dot(c[:, i, :])
        out[idx] = v[0, 0]
    return out


def fro(d):
    return math.sqrt(float(sum(x * x for x in d)))


def gamma(c):
    u = 2.0 ** -53
    return c * u / (1 - c * u)


@pytest.mark.parametrize("fmt", ["f32", "f16"])
@pytest.mark.parametrize("m,n,k,seed", [(4, 3, 2, 1), (6, 5, 3, 2), (3, 7, 4, 3)])
def test_oracle_eta_matrix_vs_exact(fmt, m, n, k, seed):
    f = W.random_factors(m, n, k, seed=seed)
    A = exact_lowrank(f.U, f.s, f.Vt)
    Ah = exact_lowrank(rnd(f.U, fmt), rnd(f.s, fmt), rnd(f.Vt, fmt))
    want = fro([A[i][j] - Ah[i][j] for i in range(m) for j in range(n)])
    got = oracle.eta_matrix(f.U, f.s, f.Vt, fmt)
    B = np.sum(np.abs(f.s) * np.linalg.norm(f.U, axis=0) * np.linalg.norm(f.Vt, axis=1))
    assert abs(got - want) <= 4 * gamma(k + 1) * B + 1e-15 * want, (got, want)


def test_oracle_eta_matrix_exact_on_dyadic_inputs():
    """12-bit dyadic factors: every product and sum of the oracle is exact,
    so only the final square root and summation round."""
    m, n, k = 5, 4, 3
    sc = 2.0 ** -12
    U = W.integer_valued((m, k), 1, -4096, 4096) * sc
    s = W.integer_valued((k,), 2, 1, 4096) * sc
    Vt = W.integer_valued((k, n), 3, -4096, 4096) * sc
    A = exact_lowrank(U, s, Vt)
    Ah = exact_lowrank(rnd(U, "f16"), rnd(s, "f16"), rnd(Vt, "f16"))
    want = fro([A[i][j] - Ah[i][j] for i in range(m) for j in range(n)])
    assert want > 0
    assert abs(oracle.eta_matrix(U, s, Vt, "f16") - want) <= 4e-16 * want


@pytest.mark.parametrize("fmt", ["f32", "f16"])
@pytest.mark.parametrize("dims,ranks", [((3, 4, 2), (1, 2, 3, 1)), ((2, 3, 2, 3), (1, 2, 2, 3, 1)),
                                        ((5, 4), (1, 3, 1))])
def test_oracle_eta_tt_vs_exact(fmt, dims, ranks):
    cores = W.make_tt(dims, ranks, "gauss", 17)
    T = exact_tt(cores)
    Th = exact_tt([rnd(c, fmt) for c in cores])
    want = fro([T[i] - Th[i] for i in T])
    got = oracle.eta_tt(cores, fmt)
    absT = float(np.linalg.norm(oracle.tt_full([np.abs(c) for c in cores])))
    assert abs(got - want) <= 4 * gamma(sum(ranks) + len(dims)) * absT + 1e-15 * want, (got, want)


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_lowrank_difference_identity_exact(fmt):
    """A - Ah = [dU, Uh] M [dV, Vh]^T with M = [[S, S], [S, dS]] holds exactly."""
    f = W.random_factors(4, 5, 3, seed=9)
    Uh, sh, Vth = rnd(f.U, fmt), rnd(f.s, fmt), rnd(f.Vt, fmt)
    U, s, Vt = F(f.U), F(f.s), F(f.Vt)
    Uhf, shf, Vhf = F(Uh), F(sh), F(Vth)
    dU, ds, dVt = U - Uhf, s - shf, Vt - Vhf
    k = 3
    Lu = np.concatenate([dU, Uhf], axis=1)
    Lv = np.concatenate([dVt.T, Vhf.T], axis=1)
    M = np.zeros((2 * k, 2 * k), dtype=object)
    M[:] = Fraction(0)
    for i in range(k):
        M[i, i] = s[i]
        M[i, k + i] = s[i]
        M[k + i, i] = s[i]
        M[k + i, k + i] = ds[i]
    D = Lu.dot(M).dot(Lv.T)
    A = exact_lowrank(f.U, f.s, f.Vt)
    Ah = exact_lowrank(Uh, sh, Vth)
    for i in range(4):
        for j in range(5):
            assert D[i, j] == A[i][j] - Ah[i][j]


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_tt_difference_recursion_exact(fmt):
    """[D_l, Zh_l] = [D_{l-1}, Zh_{l-1}] [[G_l, 0], [dG_l, Gh_l]] and
    T - Th = [D_{d-1}, Zh_{d-1}] [G_d; dG_d] hold exactly, prefix by prefix."""
    dims, ranks = (3, 2, 3, 2), (1, 2, 3, 2, 1)
    cores = W.make_tt(dims, ranks, "gauss", 23)
    G = [F(c) for c in cores]
    Gh = [F(rnd(c, fmt)) for c in cores]
    T = exact_tt(cores)
    Th = exact_tt([rnd(c, fmt) for c in cores])
    d = len(dims)
    for idx in itertools.product(*[range(x) for x in dims]):
        i0 = idx[0]
        row = np.concatenate([G[0][:, i0, :] - Gh[0][:, i0, :], Gh[0][:, i0, :]], axis=1)   # [D_1, Zh_1]
        for l in range(1, d - 1):
            g, gh = G[l][:, idx[l], :], Gh[l][:, idx[l], :]
            top = np.concatenate([g, np.full(g.shape, Fraction(0), dtype=object)], axis=1)
            bot = np.concatenate([g - gh, gh], axis=1)
            row = row.dot(np.concatenate([top, bot], axis=0))
        g, gh = G[d - 1][:, idx[d - 1], :], Gh[d - 1][:, idx[d - 1], :]
        last = np.concatenate([g, g - gh], axis=0)
        assert row.dot(last)[0, 0] == T[idx] - Th[idx]
