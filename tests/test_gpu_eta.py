"""GPU Frobenius difference (lrc_fro_diff, Sec. 5.1) and the eta / certificate
pipeline of Thm 4.1 and Thm 6.1, against the oracle."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import base_fmt, packed, to_dev

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("count", [1, 7, 8, 1000, 1_000_003, 16_777_216])
def test_fro_diff_f64_vs_oracle(lrc, cuda, count):
    a = W.gaussian((count,), count)
    b = a + W.gaussian((count,), count + 1, 1e-4)
    d, na = lrc.lrc_fro_diff(to_dev(a, cuda), "f64", to_dev(b, cuda), "f64", count)
    wd, wna = oracle.fro_diff(a, b)
    assert abs(d - wd) <= 1e-12 * wd and abs(na - wna) <= 1e-12 * wna


@pytest.mark.parametrize("fa,fb", [("f64", "f32"), ("f64", "f16"), ("f32", "f16"), ("f16", "f64")])
def test_fro_diff_mixed_formats(lrc, cuda, fa, fb):
    count = 333_333
    a64 = W.gaussian((count,), 1)
    b64 = W.gaussian((count,), 2)
    a = oracle.rounded(a64, fa)
    b = oracle.rounded(b64, fb)
    ta = to_dev(a, cuda).to(lrc.storage_dtype(fa))
    tb = to_dev(b, cuda).to(lrc.storage_dtype(fb))
    d, na = lrc.lrc_fro_diff(ta, fa, tb, fb, count)
    wd, wna = oracle.fro_diff(a, b)
    assert abs(d - wd) <= 1e-12 * wd and abs(na - wna) <= 1e-12 * wna


@pytest.mark.parametrize("lo,hi", [(-63, 63), (-62, -58), (58, 62), (-1074, -1000)])
def test_fro_diff_f64_magnitude_ranges(lrc, cuda, lo, hi):
    """Values and differences whose binary exponents straddle the limits of
    the binary32-pair squaring (|d| in [2^-48, 2^60)), binary64 subnormals,
    zeros and both signs: the sum of squares stays within 1e-12 relative."""
    rng = np.random.default_rng(lo + 2000)
    count = 400_003
    e = rng.integers(lo, hi + 1, size=count)
    a = np.ldexp(rng.uniform(0.5, 1.0, size=count), e) * rng.choice([-1.0, 1.0], size=count)
    b = a - np.ldexp(rng.uniform(0.5, 1.0, size=count), e - rng.integers(0, 3, size=count))
    a[::97] = 0.0
    b[::89] = a[::89]
    d, na = lrc.lrc_fro_diff(to_dev(a, cuda), "f64", to_dev(b, cuda), "f64", count)
    wd, wna = oracle.fro_diff(a, b)
    assert abs(d - wd) <= 1e-12 * wd and abs(na - wna) <= 1e-12 * wna


@pytest.mark.parametrize("e", [-59, -54, -49, -48, -47])
def test_fro_diff_few_small_differences(lrc, cuda, e):
    """Eight differences of one size near the lower limit of the binary32-pair
    squaring: no averaging over many elements hides a per-element error, so
    each square must be accurate to well under 1e-12 on its own."""
    rng = np.random.default_rng(50 - e)
    a = rng.uniform(0.5, 1.0, 8)
    b = a - np.ldexp(rng.uniform(0.5, 1.0, 8) * rng.choice([-1.0, 1.0], 8), e)
    d, na = lrc.lrc_fro_diff(to_dev(a, cuda), "f64", to_dev(b, cuda), "f64", 8)
    wd, wna = oracle.fro_diff(a, b)
    assert abs(d - wd) <= 1e-12 * wd and abs(na - wna) <= 1e-12 * wna


def test_fro_diff_null_b_and_determinism(lrc, cuda):
    a = to_dev(W.gaussian((5_000_001,), 9), cuda)
    r1 = lrc.lrc_fro_diff(a, "f64", None, "f64", a.numel())
    r2 = lrc.lrc_fro_diff(a, "f64", None, "f64", a.numel())
    assert r1 == r2 and r1[0] == r1[1]
    assert abs(r1[0] - oracle.fro_diff(a.cpu().numpy())[0]) <= 1e-12 * r1[0]
    z, _ = lrc.lrc_fro_diff(a, "f64", a, "f64", a.numel())
    assert z == 0.0
    # without the norm: same difference, norm not computed
    b = a * 0.5
    d1, n1 = lrc.lrc_fro_diff(a, "f64", b, "f64", a.numel())
    d2, n2 = lrc.lrc_fro_diff(a, "f64", b, "f64", a.numel(), want_norm=False)
    assert d1 == d2 and np.isnan(n2) and n1 > 0


U64_ROUNDOFF = 2.0 ** -53


def gamma(count: int) -> float:
    """gamma_m = m u / (1 - m u) of Lemma lem:dot, binary64."""
    return count * U64_ROUNDOFF / (1 - count * U64_ROUNDOFF)


def dense_f64(lrc, dev, U64, s64, Vt64):
    """A_k'^T (n x m) by the FP64 apply with identity queries."""
    m, k = U64.shape
    n = Vt64.shape[1]
    Ud, Sd, Vd = (packed(lrc, a, "f64", dev) for a in (U64, s64, Vt64))
    I = packed(lrc, np.eye(n), "f64", dev)
    Y = torch.empty((n, m), dtype=torch.float64, device=dev)
    lrc.lrc_apply(Ud, Sd, Vd, I, Y, m, n, k, n, "f64")
    return Y


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_matrix_eta_and_certificate_tiny(lrc, cuda, fmt):
    """eta_k' of the tiny workload through the GPU path: round (lrc_round_factors),
    widen (lrc_widen_factors), FP64 dense products (lrc_apply) and the
    difference (lrc_fro_diff); then Eq. matrix_condition."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    q1, sig, q2 = W.matrix_bases(cfg)
    kp = cfg.ranks[fmt]
    f = W.truncate(q1, sig, q2, kp)
    A = dense_f64(lrc, cuda, f.U, f.s, f.Vt)
    Uw = lrc.widen_matrix(packed(lrc, f.U, fmt, cuda), fmt, kp)
    Sw = lrc.widen_matrix(packed(lrc, f.s, fmt, cuda), fmt, kp)
    Vw = lrc.widen_matrix(packed(lrc, f.Vt, fmt, cuda), fmt, cfg.n)
    Ah = torch.empty_like(A)
    I = packed(lrc, np.eye(cfg.n), "f64", cuda)
    lrc.lrc_apply(Uw, Sw, Vw, I, Ah, cfg.m, cfg.n, kp, cfg.n, "f64")
    eta, nrm = lrc.lrc_fro_diff(A, "f64", Ah, "f64", A.numel())
    want = oracle.eta_matrix(f.U, f.s, f.Vt, fmt)
    # GPU and oracle evaluate A and Ahat with different rounding; by Lemma
    # lem:dot each entry is within gamma_{k+1} (|U| diag|s| |V|^T)_ij of exact,
    # for both evaluations and both matrices.
    B = np.abs(f.U) @ (np.abs(f.s)[:, None] * np.abs(f.Vt))
    tol = 4 * gamma(kp + 1) * float(np.linalg.norm(B)) + 1e-12 * want
    assert abs(eta - want) <= tol, (eta, want, tol)
    Ek = oracle.tail_error(sig, cfg.ranks["f64"])
    Ekp = oracle.tail_error(sig, kp)
    assert lrc.lrc_certified(Ek, Ekp, eta) == oracle.certified(Ek, Ekp, want) is True


@pytest.mark.parametrize("fmt", ["f32", "f16"])
def test_tt_eta(lrc, cuda, fmt):
    dims = (64, 60, 56)
    cores = W.make_tt(dims, W.capped_ranks(dims, 12), "gauss_geo", 8)
    dc = [to_dev(c, cuda).contiguous() for c in cores]
    ranks = [1] + [c.shape[2] for c in cores]
    T = torch.empty(int(np.prod(dims)), dtype=torch.float64, device=cuda)
    lrc.tt_reconstruct(dc, dims, ranks, "f64", T)
    wide = []
    for c, t in zip(cores, dc):
        flat = t.reshape(1, -1)
        p = lrc.round_matrix(flat, fmt)
        w = lrc.widen_matrix(p, fmt, flat.shape[1])[:, :flat.shape[1]].reshape(c.shape).contiguous()
        wide.append(w)
    Th = torch.empty_like(T)
    lrc.tt_reconstruct(wide, dims, ranks, "f64", Th)
    eta, _ = lrc.lrc_fro_diff(T, "f64", Th, "f64", T.numel())
    want = oracle.eta_tt(cores, fmt)
    # Sec. 5.3: entry errors are bounded by gamma |G_1(i_1)|...|G_d(i_d)|
    absT = oracle.tt_full([np.abs(c) for c in cores])
    tol = 4 * gamma(sum(ranks) + len(dims)) * float(np.linalg.norm(absT)) + 1e-12 * want
    assert abs(eta - want) <= tol, (eta, want, tol)
