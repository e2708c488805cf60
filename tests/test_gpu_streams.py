"""Per-stream library state on the GPU.  The workspace, the arrival counters
of the small-batch apply (its first kernel's last CTA per row block adds the
chunk partials) and the mapped host slot that the eta and Frobenius
reductions return their results through are kept per (device, stream): calls
interleaved on two streams give the same bits as calls on one, and
lrc_shutdown() releases all of it (the next call makes it again, zeroed)."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, oracle_inputs, packed, rel_fro

pytestmark = pytest.mark.gpu


def small_problem(lrc, dev, fmt, m, n, k, b, seed):
    f = W.random_factors(m, n, k, seed=seed)
    X = W.gaussian((b, n), seed + 1)
    ops = [packed(lrc, a, fmt, dev) for a in (f.U, f.s, f.Vt, X)]
    return f, X, ops


def as_bits(t):
    """The tensor's encodings as integers of the same width (exact compare)."""
    return t.view({2: torch.int16, 4: torch.int32, 8: torch.int64}[t.element_size()])


def apply_on(lrc, ops, shape, fmt, stream, dev):
    m, n, k, b = shape
    Y = torch.full((b, m), float("nan"), dtype=lrc.output_dtype(fmt), device=dev)
    lrc.lrc_apply(*ops, Y, m, n, k, b, fmt, stream=stream)
    return Y


@pytest.mark.parametrize("fmt,b", [("f32", 4), ("f16", 1), ("f64", 16), ("f16_o16", 3)])
def test_small_batch_apply_interleaved_on_two_streams(lrc, cuda, fmt, b):
    m, n, k = 1500, 2100, 72
    shape = (m, n, k, b)
    f, X, ops = small_problem(lrc, cuda, fmt, m, n, k, b, 31)
    ref = apply_on(lrc, ops, shape, fmt, None, cuda)
    torch.cuda.synchronize()
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    outs = []
    for i in range(6):                 # alternate the streams, several calls in flight
        st = s1 if i % 2 == 0 else s2
        with torch.cuda.stream(st):
            outs.append(apply_on(lrc, ops, shape, fmt, st, cuda))
    torch.cuda.synchronize()
    assert lrc.lrc_device_status() == 0
    for y in outs:
        assert torch.equal(as_bits(y), as_bits(ref))
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, fmt))
    assert rel_fro(ref.double().cpu().numpy(), want) <= TOL[fmt]


def test_scalar_results_on_two_streams(lrc, cuda):
    m, n, k = 900, 700, 40
    f = W.random_factors(m, n, k, seed=77)
    f64 = [packed(lrc, a, "f64", cuda) for a in (f.U, f.s, f.Vt)]
    low = [packed(lrc, a, "f16", cuda) for a in (f.U, f.s, f.Vt)]
    a = torch.from_numpy(W.gaussian((300_001,), 5)).to(cuda)
    bb = torch.from_numpy(W.gaussian((300_001,), 6)).to(cuda)
    eta0 = lrc.lrc_lowrank_eta(*f64, *low, "f16", m, n, k)
    fro0 = lrc.lrc_fro_diff(a, "f64", bb, "f64", a.numel())
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    for st in (s1, s2, s1, s2):
        with torch.cuda.stream(st):
            assert lrc.lrc_lowrank_eta(*f64, *low, "f16", m, n, k, stream=st) == eta0
            assert lrc.lrc_fro_diff(a, "f64", bb, "f64", a.numel(), stream=st) == fro0
    want = oracle.fro_diff(a.cpu().numpy(), bb.cpu().numpy())
    assert abs(fro0[0] - want[0]) <= 1e-12 * want[0] and abs(fro0[1] - want[1]) <= 1e-12 * want[1]


def test_shutdown_releases_and_calls_work_again(lrc, cuda):
    m, n, k, b = 1200, 1600, 48, 2
    shape = (m, n, k, b)
    f, X, ops = small_problem(lrc, cuda, "f32", m, n, k, b, 91)
    before = apply_on(lrc, ops, shape, "f32", None, cuda)
    a = torch.from_numpy(W.gaussian((50_000,), 8)).to(cuda)
    fro_before = lrc.lrc_fro_diff(a, "f64", None, "f64", a.numel())
    torch.cuda.synchronize()
    lrc.lrc_shutdown()
    after = apply_on(lrc, ops, shape, "f32", None, cuda)
    fro_after = lrc.lrc_fro_diff(a, "f64", None, "f64", a.numel())
    torch.cuda.synchronize()
    assert torch.equal(as_bits(before), as_bits(after))
    assert fro_after == fro_before
    assert abs(fro_after[0] - float(np.linalg.norm(a.cpu().numpy()))) <= 1e-12 * fro_after[0]
