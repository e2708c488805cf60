"""The certificate of Thm 4.1 (Eq. matrix_condition) on the hyperspectral-
shaped matrix workload, m = n = 16384, sigma_j = j^(-1.5), base rank k = 256
in FP64 against the compensated rank k' = 272.

This is the configuration whose binary16 case is designed to fail: the gain
E_256 - E_272 is about 1.6e-4 while binary16 rounding of the factors moves the
matrix by eta of about 3.3e-4, so the certificate must come out False for
binary16 and True for binary32 (the perturbation floor of Sec. 4.3 and the
failing rows of the paper's stress tables).  eta is evaluated on the GPU both
ways the library offers -- the dense route (FP64 products of the widened
factors with identity queries, then lrc_fro_diff) and the fused route
(lrc_lowrank_eta) -- and compared with the oracle's dense eta."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import packed

pytestmark = pytest.mark.gpu

CFG = W.sweep_config(1)          # m = n = 16384, ranks 256 / 272 / 272
_oracle_eta = {}


def gamma(count: int) -> float:
    u = 2.0 ** -53
    return count * u / (1 - count * u)


@pytest.fixture(scope="module")
def bases():
    return W.matrix_bases(CFG)


def oracle_eta(f, fmt):
    if fmt not in _oracle_eta:
        _oracle_eta[fmt] = oracle.eta_matrix(f.U, f.s, f.Vt, fmt)
    return _oracle_eta[fmt]


@pytest.mark.parametrize("fmt,verdict", [("f16", False), ("f32", True)])
def test_certificate_verdict_on_the_large_sweep_matrix(lrc, cuda, bases, fmt, verdict):
    q1, sig, q2 = bases
    m, n = CFG.m, CFG.n
    k, kp = CFG.ranks["f64"], CFG.ranks[fmt]
    f = W.truncate(q1, sig, q2, kp)
    want = oracle_eta(f, fmt)
    # the rank-one bound of Lemma lem:dot on every entry of both products
    tol = 4 * gamma(kp + 1) * float(np.sum(f.s)) + 1e-10 * want

    # fused route
    f64 = [packed(lrc, a, "f64", cuda) for a in (f.U, f.s, f.Vt)]
    low = [packed(lrc, a, fmt, cuda) for a in (f.U, f.s, f.Vt)]
    eta_fused, _ = lrc.lrc_lowrank_eta(*f64, *low, fmt, m, n, kp)
    assert abs(eta_fused - want) <= tol, (eta_fused, want, tol)

    # dense route: A_k'^T and Ahat_k'^T through the FP64 apply with X = I_n
    wide = [lrc.widen_matrix(low[0], fmt, kp), lrc.widen_matrix(low[1], fmt, kp),
            lrc.widen_matrix(low[2], fmt, n)]
    I = packed(lrc, np.eye(n), "f64", cuda)
    A = torch.empty((n, m), dtype=torch.float64, device=cuda)
    Ah = torch.empty_like(A)
    lrc.lrc_apply(*f64, I, A, m, n, kp, n, "f64")
    lrc.lrc_apply(*wide, I, Ah, m, n, kp, n, "f64")
    del I
    eta_dense, _ = lrc.lrc_fro_diff(A, "f64", Ah, "f64", A.numel(), want_norm=False)
    del A, Ah
    torch.cuda.empty_cache()
    assert abs(eta_dense - want) <= tol, (eta_dense, want, tol)

    Ek, Ekp = oracle.tail_error(sig, k), oracle.tail_error(sig, kp)
    assert oracle.certified(Ek, Ekp, want) is verdict
    assert lrc.lrc_certified(Ek, Ekp, eta_fused) is verdict
    assert lrc.lrc_certified(Ek, Ekp, eta_dense) is verdict
    if fmt == "f16":
        # the designed margin: eta is about twice the gain E_k - E_k'
        assert want > 1.5 * (Ek - Ekp)
