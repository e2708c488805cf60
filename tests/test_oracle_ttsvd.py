"""Pins for the oracle's factorization side: TT-SVD (Sec. 5; Alg.
alg:tt_compensation steps 1-2) and the left-orthogonal gauge (Sec. 6.1).

- The paper's printed errors: TT-SVD of hilbert_3d (100^3) and decay_3d
  (60^3), the closed-form tensors of Sec. 7.2, at the base ranks of Table
  tab:tt_three_way_detail reproduces its E_R column, and at the augmented
  ranks (whose FP32 rounding perturbation is far below the error) its
  FP32 error column (tests/golden/tt_three_way.csv).
- d = 2: TT-SVD is the truncated SVD, so its error is the Eckart-Young tail.
- Known-rank tensors are recovered exactly at their ranks.
- The error identity ||T - T_R||^2 = sum of the discarded s^2.
- Left-orthogonalization leaves the tensor unchanged and makes cores
  1..d-1 orthonormal, with ||G_d|| = ||T||."""
import csv
import math
import os

import numpy as np
import pytest

import oracle
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def golden_rows():
    with open(os.path.join(GOLDEN, "tt_three_way.csv")) as fh:
        return [r for r in csv.reader(l for l in fh if not l.startswith("#"))]


def rel_err(T, cores):
    return oracle.fro_diff(T.reshape(-1), oracle.tt_full(cores).reshape(-1))[0] / oracle.fro_diff(T)[0]


@pytest.fixture(scope="module")
def tensors():
    return {"hilbert_3d": W.hilbert_3d(100), "decay_3d": W.decay_3d(60)}


def test_printed_base_errors(tensors):
    seen = set()
    for name, R, Rp, prec, e_r, new, eta, *_ in golden_rows():
        if (name, R) in seen:
            continue
        seen.add((name, R))
        T = tensors[name]
        R = int(R)
        cores, delta2 = oracle.tt_svd(T, (1, R, R, 1))
        e = rel_err(T, cores)
        assert abs(e - float(e_r)) <= 0.005 * float(e_r), (name, R, e, e_r)
        # the error identity of TT-SVD
        nT = oracle.fro_diff(T)[0]
        assert abs(math.sqrt(sum(delta2)) / nT - e) <= 1e-6 * e + 1e-15, (name, R)
    assert len(seen) == 6


def test_printed_augmented_errors_fp32(tensors):
    """FP32 rows whose perturbation eta is at least 100x below the printed
    new error: that error is the FP64 augmented error E_{R+} to 3 digits."""
    n = 0
    for name, R, Rp, prec, e_r, new, eta, *_ in golden_rows():
        if prec != "FP32" or float(eta) * 100 > float(new):
            continue
        T = tensors[name]
        cores, _ = oracle.tt_svd(T, (1, int(Rp), int(Rp), 1))
        e = rel_err(T, cores)
        assert abs(e - float(new)) <= 0.006 * float(new), (name, Rp, e, new)
        n += 1
    assert n >= 7


def test_two_way_is_eckart_young():
    A = W.gaussian((40, 25), 3) @ np.diag(np.exp(-0.3 * np.arange(25))) @ W.gaussian((25, 33), 4)
    s = np.linalg.svd(A, compute_uv=False)
    for r in (1, 5, 12, 25):
        cores, delta2 = oracle.tt_svd(A, (1, r, 1))
        tail = math.fsum((s[r:] ** 2)[::-1])
        # singular values past the rank are rounding noise of size u s_1
        assert abs(delta2[0] - tail) <= 1e-12 * tail + 1e-26 * s[0] ** 2
        err = oracle.fro_diff(A.reshape(-1), oracle.tt_full(cores).reshape(-1))[0]
        assert abs(err ** 2 - tail) <= 1e-10 * tail + 1e-26 * s[0] ** 2 * A.size


@pytest.mark.parametrize("dims,ranks", [((7, 9, 8), (1, 3, 4, 1)), ((5, 6, 4, 7), (1, 2, 5, 3, 1)),
                                        ((30, 31, 32), (1, 6, 5, 1))])
def test_exact_recovery_of_known_rank_tensors(dims, ranks):
    T = oracle.tt_full(W.make_tt(dims, ranks, "gauss_geo", 5))
    cores, delta2 = oracle.tt_svd(T, ranks)
    assert rel_err(T, cores) <= 1e-13
    assert math.sqrt(sum(delta2)) <= 1e-13 * oracle.fro_diff(T)[0]
    assert [c.shape[2] for c in cores[:-1]] == list(ranks[1:-1])


def test_sum_of_functions_has_rank_two():
    f = [np.cos(np.arange(n) * 0.3 + l) for l, n in enumerate((11, 12, 13))]
    T = f[0][:, None, None] + f[1][None, :, None] + f[2][None, None, :]
    cores, delta2 = oracle.tt_svd(T, (1, 2, 2, 1))
    assert rel_err(T, cores) <= 1e-13
    _, d1 = oracle.tt_svd(T, (1, 1, 1, 1))
    assert sum(d1) > 1e-3 * oracle.fro_diff(T)[0] ** 2     # rank 1 is not enough


def test_left_orthogonalize_invariants():
    dims, ranks = (9, 8, 7, 6), (1, 5, 6, 4, 1)
    cores = [W.gaussian((ranks[l], dims[l], ranks[l + 1]), 40 + l) for l in range(4)]
    T = oracle.tt_full(cores)
    lo = oracle.tt_left_orthogonalize(cores)
    assert oracle.fro_diff(T.reshape(-1), oracle.tt_full(lo).reshape(-1))[0] <= 1e-13 * oracle.fro_diff(T)[0]
    for c in lo[:-1]:
        Q = c.reshape(-1, c.shape[2])
        assert np.allclose(Q.T @ Q, np.eye(Q.shape[1]), atol=1e-14)
    assert abs(oracle.fro_diff(lo[-1])[0] - oracle.fro_diff(T)[0]) <= 1e-13 * oracle.fro_diff(T)[0]
    # TT-SVD already returns left-orthonormal cores (Sec. 7.2)
    svd_cores, _ = oracle.tt_svd(T, ranks)
    for c in svd_cores[:-1]:
        Q = c.reshape(-1, c.shape[2])
        assert np.allclose(Q.T @ Q, np.eye(Q.shape[1]), atol=1e-13)
