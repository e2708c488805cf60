"""Pins for the oracle's certificate and storage accounting against the
values the paper prints.

Fixtures under tests/golden/ are transcriptions of the paper's tables, each
file citing its table.  Printed values carry three significant digits, so
every comparison allows the printing slack.
"""
import csv
import math
import os

import numpy as np
import pytest

import oracle
import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
PREC = {"FP64": "f64", "FP32": "f32", "FP16": "f16"}
SLACK = 0.005          # half a unit in the third significant digit


def rows(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return [r for r in csv.reader(l for l in fh if not l.startswith("#"))]


def verdict_consistent(e_base, new_err, eta, printed_yes):
    """The paper's verdict is E_aug + eta <= E_base (Eq. matrix_condition /
    Eq. tt_condition) with the unprinted E_aug bounded by the triangle
    inequality |new - E_aug| <= eta.  Check, through the oracle's predicate,
    that some printing-consistent E_aug gives the printed verdict."""
    lo, hi = 1 - SLACK, 1 + SLACK
    if printed_yes:
        return oracle.certified(e_base * hi, new_err * lo - eta * lo, eta * lo)
    return not oracle.certified(e_base * lo, new_err * hi + eta * hi, eta * hi)


def test_matrix_speed_storage_ratios():
    for method, prec, rank, ratio in rows("matrix_speed_storage.csv"):
        got = oracle.matrix_storage_ratio(1000, 700, 40, int(rank), PREC[prec])
        assert abs(got - float(ratio)) <= 5e-5 + 1e-12, method


def test_tail_stress_storage_and_verdicts():
    n_yes = n_no = 0
    for name, k, k1, ek, eta, new, ratio, storage, cert in rows("tail_stress_fp16.csv"):
        got = 100 * oracle.matrix_storage_ratio(494, 494, int(k), int(k1), "f16")
        assert abs(got - float(storage)) <= 0.05 + 1e-9, (name, k)
        yes = cert == "Yes"
        assert verdict_consistent(float(ek), float(new), float(eta), yes), (name, k)
        n_yes += yes
        n_no += not yes
    assert n_yes == 10 and n_no == 7


@pytest.mark.parametrize("fixture,dims", [
    ("tt_three_way.csv", {"decay_3d": (60,) * 3, "hilbert_3d": (100,) * 3}),
    ("tt_six_way.csv", {"decay_6d": (12,) * 6, "hilbert_6d": (12,) * 6}),
])
def test_tt_storage_ratios_and_verdicts(fixture, dims):
    for name, R, Rp, prec, er, new, eta, eratio, mratio, cert in rows(fixture):
        dd = dims[name]
        base = W.capped_ranks(dd, int(R))
        aug = W.capped_ranks(dd, int(Rp))
        got = oracle.tt_storage_ratio(dd, base, aug, PREC[prec])
        assert abs(got - float(mratio)) <= 0.005 + 1e-9, (name, R, Rp, prec, got)
        assert verdict_consistent(float(er), float(new), float(eta), cert == "Yes"), (name, R, Rp, prec)


def test_tt_storage_three_core_closed_form():
    # Sec. 6.1: for a uniform three-core TT the exact ratio is
    # (b/64) (R+delta)(R+delta+2) / (R (R+2))
    for R, delta, fmt in [(4, 1, "f16"), (16, 4, "f32"), (8, 4, "f16"), (32, 4, "f32")]:
        dd = (200, 200, 200)
        got = oracle.tt_storage_ratio(dd, (1, R, R, 1), (1, R + delta, R + delta, 1), fmt)
        b = oracle.BITS[fmt]
        want = b / 64 * (R + delta) * (R + delta + 2) / (R * (R + 2))
        assert abs(got - want) <= 1e-15


def test_hyperspectral_storage_and_memory_matched_rank():
    mib = 2.0 ** 20
    budgets = {}
    for name, n1, n2, n3, r, prec, st in rows("hyperspectral_storage.csv"):
        dd = (int(n1), int(n2), int(n3))
        got = oracle.tt_storage_bits(dd, W.capped_ranks(dd, int(r)), PREC[prec]) / 8 / mib
        assert abs(got - float(st)) <= 0.005 + 1e-9, (name, prec)
        if prec == "FP16":
            budgets[name] = (dd, got * 8 * mib)
    # Sec. 8: the largest FP64 uniform rank within each FP16 (36,36) budget is (17,17)
    for name, (dd, budget) in budgets.items():
        best = max(R for R in range(1, 64)
                   if oracle.tt_storage_bits(dd, W.capped_ranks(dd, R), "f64") <= budget)
        assert best == 17, name


def test_public_tensor_verdicts():
    for case, er, eta, new, ratio, cert in rows("public_tt_failures.csv"):
        assert verdict_consistent(float(er), float(new), float(eta), cert == "Yes"), case
        assert abs(float(new) / float(er) - float(ratio)) <= 0.02


def test_squared_form_equivalence():
    """Thm 4.1: E_{k+1} + eta <= E_k  <=>  eta <= E_k and
    sigma_{k+1}^2 >= 2 eta E_k - eta^2, with E_{k+1}^2 = E_k^2 - sigma_{k+1}^2."""
    rng = np.random.default_rng(4)
    agree = 0
    for _ in range(5000):
        ek = float(rng.uniform(1e-3, 1.0))
        ek1 = ek * float(rng.uniform(0.0, 1.0))
        eta = ek * float(rng.uniform(0.0, 1.5))
        sig2 = ek * ek - ek1 * ek1
        lhs = oracle.certified(ek, ek1, eta)
        margin = abs(ek1 + eta - ek)
        if margin < 1e-9:
            continue
        rhs = (eta <= ek) and (sig2 >= 2 * eta * ek - eta * eta)
        assert lhs == rhs
        agree += 1
    assert agree > 4900


def test_paper_rank_capping_example():
    # Sec. 7.4: Salinas-A (83 x 86 x 204) at nominal rank 160 gives R = (83, 160)
    assert W.capped_ranks((83, 86, 204), 160) == (1, 83, 160, 1)
    assert W.capped_ranks((83, 86, 204), 161) == (1, 83, 161, 1)


def test_matrix_bound_pinned_to_eckart_young_equality():
    """Thm 4.1 Eq. matrix_universal_bound at its equality case.  With eta = 0
    the compensated factors are the exact rank-(k+1) truncation, whose error is
    E_{k+1} = (E_k^2 - sigma_{k+1}^2)^(1/2) (Sec. 4, Eckart-Young), so the
    bound must equal (i) the oracle's tail error at k + 1, (ii) the closed-form
    geometric tail of the tiny workload's spectrum sigma_j = 2^(-j/16), and
    (iii) the dense error ||A - A_{k+1}||_F itself; and it must grow with eta
    at unit slope.  A dropped square root, a + in place of the -, the wrong
    sigma index or a scaled eta each fail one of these."""
    cfg = W.MATRIX_CONFIGS["tiny"]
    q1, sig, q2 = W.matrix_bases(cfg, k_max=512)
    ln2 = math.log(2.0)

    def geo_tail(k):   # (sum_{j=k+1}^{512} 2^(-j/8))^(1/2), 1-based j
        t2 = math.exp2(-(k + 1) / 8.0) * -math.expm1(-(512 - k) / 8.0 * ln2) / -math.expm1(-ln2 / 8.0)
        return math.sqrt(t2)

    for k in (0, 1, 31, 32, 33, 100, 255, 400, 510):
        ek = oracle.tail_error(sig, k)
        b0 = oracle.matrix_bound(ek, sig[k], 0.0)             # sig[k] = sigma_{k+1}
        e_next = oracle.tail_error(sig, k + 1)
        assert abs(b0 - e_next) <= 1e-14 * e_next, k
        # closed form, with E_k also taken from the closed form
        b0c = oracle.matrix_bound(geo_tail(k), math.exp2(-(k + 1) / 16.0), 0.0)
        assert abs(b0c - geo_tail(k + 1)) <= 1e-13 * geo_tail(k + 1), k
        for eta in (1e-9, 3.7e-4, 0.25):
            assert abs(oracle.matrix_bound(ek, sig[k], eta) - (b0 + eta)) <= 1e-15 * (b0 + eta), (k, eta)
    # (iii) the bound is attained: ||A - A_{k+1}||_F from the dense oracle products
    A_T = (q2 * sig) @ q1.T
    for k in (31, 32, 33):
        f = W.truncate(q1, sig, q2, k + 1)
        err, _ = oracle.fro_diff(A_T, oracle.apply(f.U, f.s, f.Vt, np.eye(512)))
        b0 = oracle.matrix_bound(oracle.tail_error(sig, k), sig[k], 0.0)
        assert abs(err - b0) <= 1e-12 * b0, k
