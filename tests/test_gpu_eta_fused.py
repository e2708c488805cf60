"""Fused eta without dense reconstruction (lrc_lowrank_eta, lrc_tt_eta; the
eta of Thm 4.1 and eta_TT of Thm 6.1) against the oracle's dense definition
(both products formed in FP64, Frobenius norm of the difference).

Tolerances.  The oracle forms every entry of A and Ahat with a sum of k + 1
rounded products, so by Lemma lem:dot each entry is within
gamma_{k+1} (|U| diag|s| |V|^T)_ij of its exact value; the Frobenius norm of
that bound is at most sum_l |s_l| ||u_l|| ||v_l|| (one rank-one term per l).
The fused path carries the rounding errors explicitly and is far more
accurate than that, so the bar is the oracle's own bound plus 1e-10 eta.
On dyadic inputs with few significant bits every product and sum of the
oracle is exact, and the bar tightens to 1e-12 relative."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import base_fmt, packed, to_dev

pytestmark = pytest.mark.gpu

FMTS = ["f64", "f32", "f16", "f16_o16"]


def gamma(count: int) -> float:
    u = 2.0 ** -53
    return count * u / (1 - count * u)


def rank_one_bound(U, s, Vt) -> float:
    return float(np.sum(np.abs(s) * np.linalg.norm(U, axis=0) * np.linalg.norm(Vt, axis=1)))


def fused_matrix(lrc, dev, U, s, Vt, fmt, **kw):
    m, k = U.shape
    n = Vt.shape[1]
    f64 = [packed(lrc, a, "f64", dev) for a in (U, s, Vt)]
    low = [packed(lrc, a, fmt, dev) for a in (U, s, Vt)]
    return lrc.lrc_lowrank_eta(*f64, *low, fmt, m, n, k, **kw)


def check_matrix(lrc, dev, U, s, Vt, fmt, exact=False):
    eta, nrm = fused_matrix(lrc, dev, U, s, Vt, fmt)
    if fmt == "f64":
        assert eta == 0.0
        return eta
    want = oracle.eta_matrix(U, s, Vt, base_fmt(fmt))
    k = U.shape[1]
    tol = (1e-12 * want) if exact else (4 * gamma(k + 1) * rank_one_bound(U, s, Vt) + 1e-10 * want)
    assert abs(eta - want) <= tol, (eta, want, tol)
    return eta


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("m,n,k", [(1, 1, 1), (5, 4, 3), (37, 29, 7), (300, 200, 33), (1000, 777, 144),
                                   (129, 1500, 17)])
def test_lowrank_eta_vs_oracle(lrc, cuda, fmt, m, n, k):
    f = W.random_factors(m, n, k, seed=m * 7 + n + k)
    check_matrix(lrc, cuda, f.U, f.s, f.Vt, fmt)


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_lowrank_eta_tiny_workload(lrc, cuda, fmt):
    """The 512 x 512 workload at k' = 33 / 34 (sigma_j = 2^(-j/16)); the
    certificate of Eq. matrix_condition holds with the fused eta."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    q1, sig, q2 = W.matrix_bases(cfg)
    kp = cfg.ranks[fmt]
    f = W.truncate(q1, sig, q2, kp)
    eta = check_matrix(lrc, cuda, f.U, f.s, f.Vt, fmt)
    Ek = oracle.tail_error(sig, cfg.ranks["f64"])
    Ekp = oracle.tail_error(sig, kp)
    assert lrc.lrc_certified(Ek, Ekp, eta)


@pytest.mark.parametrize("m,n,k", [(70, 45, 5), (300, 260, 20)])
def test_lowrank_eta_dyadic_f16_exact(lrc, cuda, m, n, k):
    """13-bit dyadic factors: binary16 rounds most entries, and every product
    and sum of the oracle is exact."""
    sc = 2.0 ** -12
    U = W.integer_valued((m, k), 11, -4096, 4096) * sc
    s = W.integer_valued((k,), 12, 1, 4096) * sc
    Vt = W.integer_valued((k, n), 13, -4096, 4096) * sc
    for fmt in ("f16", "f16_o16"):
        check_matrix(lrc, cuda, U, s, Vt, fmt, exact=True)


@pytest.mark.parametrize("side", ["U", "V"])
def test_lowrank_eta_dyadic_f32_exact(lrc, cuda, side):
    """25-bit dyadic entries in one factor (binary32 rounds them), 8-bit in
    the others (kept exactly): the oracle is exact, one error term at a time."""
    m, n, k = 90, 70, 6
    big = 2.0 ** -24
    small = 2.0 ** -7
    U = W.integer_valued((m, k), 21, -(1 << 24), 1 << 24) * big if side == "U" else \
        W.integer_valued((m, k), 21, -128, 128) * small
    Vt = W.integer_valued((k, n), 22, -(1 << 24), 1 << 24) * big if side == "V" else \
        W.integer_valued((k, n), 22, -128, 128) * small
    s = W.integer_valued((k,), 23, 1, 128) * small
    check_matrix(lrc, cuda, U, s, Vt, "f32", exact=True)


def test_lowrank_eta_norm_and_determinism(lrc, cuda):
    """norm_out is ||U diag(s) V^T||_F = ||s||_2 for orthonormal U, V; two
    calls give identical bits; want_norm=False leaves the norm out."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    q1, sig, q2 = W.matrix_bases(cfg)
    f = W.truncate(q1, sig, q2, 34)
    r1 = fused_matrix(lrc, cuda, f.U, f.s, f.Vt, "f16")
    r2 = fused_matrix(lrc, cuda, f.U, f.s, f.Vt, "f16")
    assert r1 == r2
    assert abs(r1[1] - float(np.linalg.norm(f.s))) <= 1e-13 * r1[1]
    e3, n3 = fused_matrix(lrc, cuda, f.U, f.s, f.Vt, "f16", want_norm=False)
    assert e3 == r1[0] and np.isnan(n3)


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_lowrank_eta_large_workload(lrc, cuda, fmt):
    """m = 16384, n = 8192, k' = 136 / 144, sigma_j = j^(-1.5): the full-size
    launch, against the oracle's full dense eta."""
    cfg = W.MATRIX_CONFIGS["large"]
    q1, sig, q2 = W.matrix_bases(cfg)
    f = W.truncate(q1, sig, q2, cfg.ranks[fmt])
    eta = check_matrix(lrc, cuda, f.U, f.s, f.Vt, fmt)
    Ek = oracle.tail_error(sig, cfg.ranks["f64"])
    Ekp = oracle.tail_error(sig, cfg.ranks[fmt])
    assert lrc.lrc_certified(Ek, Ekp, eta) == oracle.certified(Ek, Ekp, eta)


def test_lowrank_eta_row_blocks_add_up(lrc, cuda):
    """eta^2 is additive over row blocks of U: the full launch of the
    16384 x 16384, k' = 272 sweep factors equals the sum over four blocks."""
    cfg = W.sweep_config(4096)
    f = W.matrix_factors(cfg, "f16")
    m = f.U.shape[0]
    full, _ = fused_matrix(lrc, cuda, f.U, f.s, f.Vt, "f16")
    parts = [fused_matrix(lrc, cuda, f.U[a:a + m // 4], f.s, f.Vt, "f16")[0] for a in range(0, m, m // 4)]
    assert abs(full ** 2 - sum(p * p for p in parts)) <= 1e-11 * full ** 2
    # and one block against the oracle, evaluated on the transpose (eta is
    # the same for A^T; the oracle's dense product then runs over 256 columns)
    blk = f.U[: m // 64]
    want = oracle.eta_matrix(np.ascontiguousarray(f.Vt.T), f.s, np.ascontiguousarray(blk.T), "f16")
    got, _ = fused_matrix(lrc, cuda, blk, f.s, f.Vt, "f16")
    assert abs(got - want) <= 4 * gamma(f.U.shape[1] + 1) * rank_one_bound(blk, f.s, f.Vt) + 1e-10 * want


# ---------------------------------------------------------------------------
# Tensor Train
# ---------------------------------------------------------------------------

def fused_tt(lrc, dev, cores, fmt, **kw):
    dims = [c.shape[1] for c in cores]
    ranks = [1] + [c.shape[2] for c in cores]
    c64 = [to_dev(c, dev).contiguous() for c in cores]
    low = []
    for t in c64:
        flat = t.reshape(1, -1)
        p = lrc.round_matrix(flat, fmt)
        low.append(p[:, :flat.shape[1]].reshape(t.shape).contiguous())
    return lrc.lrc_tt_eta(c64, low, dims, ranks, fmt, **kw)


def check_tt(lrc, dev, cores, fmt, exact=False):
    eta, nrm = fused_tt(lrc, dev, cores, fmt)
    if fmt == "f64":
        assert eta == 0.0
        return eta, nrm
    want = oracle.eta_tt(cores, base_fmt(fmt))
    ranks = [1] + [c.shape[2] for c in cores]
    if exact:
        tol = 1e-12 * want
    else:
        absT = float(np.linalg.norm(oracle.tt_full([np.abs(c) for c in cores])))
        tol = 4 * gamma(sum(ranks) + len(cores)) * absT + 1e-10 * want
    assert abs(eta - want) <= tol, (eta, want, tol)
    return eta, nrm


TT_SHAPES = [
    ((37, 29), (1, 5, 1)),
    ((7, 9, 11), (1, 3, 4, 1)),
    ((64, 60, 56), W.capped_ranks((64, 60, 56), 12)),
    ((5, 6, 7, 8), (1, 4, 9, 6, 1)),
    ((4,) * 6, (1, 4, 8, 8, 8, 4, 1)),
    ((3, 16, 16), (1, 3, 16, 1)),
    ((300, 2, 40), (1, 33, 17, 1)),
]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("dims,ranks", TT_SHAPES)
def test_tt_eta_vs_oracle(lrc, cuda, fmt, dims, ranks):
    cores = W.make_tt(dims, ranks, "gauss_geo", 5 + sum(dims))
    check_tt(lrc, cuda, cores, fmt)


def test_tt_eta_dyadic_exact(lrc, cuda):
    """12-bit dyadic cores: binary16 rounds them and the oracle's chain is exact."""
    dims, ranks = (6, 7, 5), (1, 3, 4, 1)
    sc = 2.0 ** -11
    cores = [W.integer_valued((ranks[l], dims[l], ranks[l + 1]), 40 + l, -2048, 2048) * sc for l in range(3)]
    check_tt(lrc, cuda, cores, "f16", exact=True)


@pytest.mark.parametrize("name", ["tt3", "tt6"])
@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_tt_eta_full_workloads(lrc, cuda, name, fmt):
    """The 256^3 and 16^6 workloads at their compensated ranks."""
    cfg = W.TT_CONFIGS[name]
    cores = W.tt_cores(cfg, fmt)
    eta, nrm = check_tt(lrc, cuda, cores, fmt)
    T = oracle.tt_full(cores)
    assert abs(nrm - float(np.linalg.norm(T))) <= 1e-12 * nrm


def test_tt_eta_hyperspectral_first_mode_blocks(lrc, cuda):
    """512 x 512 x 224 at ranks (1,70,52,1): eta_TT^2 is additive over blocks
    of i_1 (rows of G_1); the full launch equals the sum of four blocks and
    one block matches the oracle."""
    cfg = W.TT_CONFIGS["tt_hsi"]
    cores = W.tt_cores(cfg, "f16")
    full, _ = fused_tt(lrc, cuda, cores, "f16")
    n1 = cores[0].shape[1]
    parts = []
    for a in range(0, n1, n1 // 4):
        sub = [np.ascontiguousarray(cores[0][:, a:a + n1 // 4, :])] + cores[1:]
        parts.append(fused_tt(lrc, cuda, sub, "f16")[0])
    assert abs(full ** 2 - sum(p * p for p in parts)) <= 1e-11 * full ** 2
    sub = [np.ascontiguousarray(cores[0][:, :8, :])] + cores[1:]
    check_tt(lrc, cuda, sub, "f16")


def test_tt_eta_determinism(lrc, cuda):
    cores = W.tt_cores(W.TT_CONFIGS["tt3"], "f16")
    assert fused_tt(lrc, cuda, cores, "f16") == fused_tt(lrc, cuda, cores, "f16")
