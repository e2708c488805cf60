"""Failure detection without a GPU fault: a bounded device wait that runs out
is reported as LRC_ERR_TIMEOUT by lrc_device_status, and the context stays
usable afterwards."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, oracle_inputs, packed, rel_fro

pytestmark = pytest.mark.gpu


def test_wait_timeout_is_reported_and_context_survives(lrc, cuda):
    assert lrc.lrc_device_status() == 0
    lrc.lrc_selftest_wait_timeout(1_000_000)          # 1 ms wait on a barrier nobody arrives on
    assert lrc.lrc_device_status() == -6
    assert lrc.lrc_device_status() == 0               # the error word was cleared
    # the device still computes correctly
    f = W.random_factors(300, 200, 40, seed=1)
    X = W.gaussian((130, 200), 2)
    Ud, Sd, Vd, Xd = (packed(lrc, a, "f16", cuda) for a in (f.U, f.s, f.Vt, X))
    Y = torch.empty((130, 300), dtype=torch.float32, device=cuda)
    lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, 300, 200, 40, 130, "f16")
    assert lrc.lrc_device_status() == 0
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, "f16"))
    assert rel_fro(Y.double().cpu().numpy(), want) <= TOL["f16"]


def test_selftest_rejects_bad_limit(lrc, cuda):
    with pytest.raises(lrc.LrcError):
        lrc.lrc_selftest_wait_timeout(0)
