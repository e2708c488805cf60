"""Pins for the oracle's matrix apply (Sec. 4.4, Eq. gpu_matrix_apply), its
Frobenius difference (Sec. 5.1) and the eta of Thm 4.1.

Independent facts used: exact integer arithmetic (pure Python ints), the
Eckart-Young identity E_k^2 = sum_{j>k} sigma_j^2 with a closed-form
geometric tail, numpy/LAPACK matrix products, math.fsum, and the paper's
printed eta magnitudes relative to the unit roundoff.
"""
import math

import numpy as np
import pytest

import oracle
import workloads as W


def brute_apply_int(U, s, Vt, X):
    """Exact integer evaluation with Python ints: Y[c,r] = sum_j U[r,j] s_j sum_i X[c,i] Vt[j,i]."""
    m, k = U.shape
    n = Vt.shape[1]
    b = X.shape[0]
    Ui = [[int(v) for v in row] for row in U]
    Vi = [[int(v) for v in row] for row in Vt]
    Xi = [[int(v) for v in row] for row in X]
    si = [int(v) for v in s]
    Y = np.zeros((b, m))
    for c in range(b):
        w = [si[j] * sum(Xi[c][i] * Vi[j][i] for i in range(n)) for j in range(k)]
        for r in range(m):
            Y[c, r] = float(sum(w[j] * Ui[r][j] for j in range(k)))
    return Y


@pytest.mark.parametrize("m,n,k,b", [(7, 5, 3, 4), (5, 9, 6, 1), (13, 11, 1, 3), (4, 4, 4, 4)])
def test_apply_exact_on_integer_inputs(m, n, k, b):
    U = W.integer_valued((m, k), 1)
    s = W.integer_valued((k,), 2, 1, 5)
    Vt = W.integer_valued((k, n), 3)
    X = W.integer_valued((b, n), 4)
    assert np.array_equal(oracle.apply(U, s, Vt, X), brute_apply_int(U, s, Vt, X))


def test_apply_matches_numpy_products():
    f = W.random_factors(37, 29, 11, seed=5)
    X = W.gaussian((6, 29), 6)
    want = ((X @ f.Vt.T) * f.s) @ f.U.T
    got = oracle.apply(f.U, f.s, f.Vt, X)
    assert np.max(np.abs(got - want)) <= 1e-14 * np.max(np.abs(want))
    rows = [5, 0, 3]
    assert np.array_equal(oracle.apply_rows(f.U, f.s, f.Vt, X, rows), got[rows])


def test_apply_identity_queries_give_dense_transpose():
    # X = I_n gives Y = V diag(s) U^T = A_k^T
    f = W.random_factors(9, 6, 4, seed=8)
    A = f.U @ np.diag(f.s) @ f.Vt
    Y = oracle.apply(f.U, f.s, f.Vt, np.eye(6))
    assert np.allclose(Y, A.T, rtol=0, atol=1e-15)


def test_eckart_young_identity_tiny_config():
    """Sec. 4: ||A - A_k||_F^2 = sum_{j>k} sigma_j^2 for A = Q1 diag(sigma) Q2^T,
    sigma_j = 2^(-j/16), m = n = 512 (the tiny workload)."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    q1, sig, q2 = W.matrix_bases(cfg, k_max=512)
    A_T = (q2 * sig) @ q1.T                      # A^T, built with numpy
    for k in (1, 32, 33, 34, 256):
        f = W.truncate(q1, sig, q2, k)
        Yk = oracle.apply(f.U, f.s, f.Vt, np.eye(512))   # A_k^T
        err, _ = oracle.fro_diff(A_T, Yk)
        # closed-form geometric tail: sum_{j=k+1}^{512} 2^(-j/8)
        tail2 = (math.exp2(-(k + 1) / 8.0) * -math.expm1(-(512 - k) / 8.0 * math.log(2.0))
                 / -math.expm1(-math.log(2.0) / 8.0))
        assert abs(err ** 2 - tail2) <= 1e-12 * tail2, k
        assert abs(oracle.tail_error(sig, k) - math.sqrt(tail2)) <= 1e-13 * math.sqrt(tail2)
    # the printed-to-6-digits values of this spectrum
    assert abs(oracle.tail_error(sig, 0) - 3.32397) < 5e-6
    assert abs(oracle.tail_error(sig, 32) - 0.830993) < 5e-7
    assert abs(oracle.tail_error(sig, 34) - 0.762024) < 5e-7


def test_fro_diff_basic_facts():
    a = np.full(1000, 3.0)
    d, na = oracle.fro_diff(a, a)
    assert d == 0.0 and abs(na - 3.0 * math.sqrt(1000)) < 1e-12
    d, _ = oracle.fro_diff(a, None)
    assert abs(d - 3.0 * math.sqrt(1000)) < 1e-12
    # compensated sum: squares exact in binary64, compare against math.fsum
    rng = np.random.default_rng(1)
    x = rng.integers(-2 ** 20, 2 ** 20, 100_000).astype(np.float64) * 2.0 ** -10
    x[0] = 2.0 ** 26                                # one dominant term
    d, _ = oracle.fro_diff(x)
    exact = math.sqrt(math.fsum(v * v for v in x))
    assert abs(d - exact) <= 1e-15 * exact
    # difference is taken element-wise before squaring
    y = x + 0.5
    d, _ = oracle.fro_diff(y, x)
    assert abs(d - 0.5 * math.sqrt(x.size)) < 1e-12


def test_eta_magnitude_matches_paper_scale():
    """Relative eta of rounded orthonormal factors sits near 0.7 u: the paper
    prints FP16 eta of 2.2e-4..6.4e-4 and FP32 eta of 3.7e-8..7.9e-8 relative
    to the norm (Tables tab:tail_stress_detailed, tab:tt_three_way_detail,
    tab:synthetic_tt_d6_detail, tab:public_tensor_detail_errors)."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    for fmt in ("f32", "f16"):
        f = W.matrix_factors(cfg, fmt)
        eta = oracle.eta_matrix(f.U, f.s, f.Vt, fmt)
        nrm = math.sqrt(float(np.sum(f.s ** 2)))
        ratio = eta / (oracle.UNIT_ROUNDOFF[fmt] * nrm)
        assert 0.6 <= ratio <= 0.8, (fmt, ratio)
        rel = eta / nrm
        lo, hi = {"f16": (2.1e-4, 6.4e-4), "f32": (3.7e-8, 7.9e-8)}[fmt]
        assert lo <= rel <= hi


def test_certificate_triangle_bounds_random_cases():
    """Thm 4.1: |E_k' - eta| <= ||A - Ahat_k'||_F <= E_k' + eta, and the
    certificate E_k' + eta <= E_k implies ||A - Ahat_k'||_F <= E_k."""
    rng = np.random.default_rng(11)
    n_cert = 0
    for case in range(200):
        m = int(rng.integers(8, 40))
        n = int(rng.integers(8, 40))
        p = min(m, n)
        k = int(rng.integers(1, p - 1))
        kp = int(rng.integers(k + 1, p + 1))
        fmt = ("f32", "f16")[case % 2]
        decay = float(rng.uniform(0.05, 3.0))
        sig = np.sort(rng.uniform(0.1, 1.0, p) * np.exp(-decay * np.arange(p)))[::-1]
        if case % 5 == 0:
            sig = np.maximum(sig, 1e-2)               # flat tail: near the FP16 floor
        q1 = W.orthonormal_columns(m, p, 10_000 + case)
        q2 = W.orthonormal_columns(n, p, 20_000 + case)
        A_T = (q2 * sig) @ q1.T
        f = W.truncate(q1, sig, q2, kp)
        Ah = oracle.apply(oracle.rounded(f.U, fmt), oracle.rounded(f.s, fmt),
                          oracle.rounded(f.Vt, fmt), np.eye(n))
        new_err, _ = oracle.fro_diff(A_T, Ah)
        eta = oracle.eta_matrix(f.U, f.s, f.Vt, fmt)
        Ek, Ekp = oracle.tail_error(sig, k), oracle.tail_error(sig, kp)
        tol = 1e-13 * max(1.0, Ek)
        assert abs(Ekp - eta) <= new_err + tol
        assert new_err <= Ekp + eta + tol
        if kp == k + 1:
            assert new_err <= oracle.matrix_bound(Ek, sig[k], eta) + tol
        if oracle.certified(Ek, Ekp, eta):
            n_cert += 1
            assert new_err <= Ek + tol
    assert n_cert > 50
