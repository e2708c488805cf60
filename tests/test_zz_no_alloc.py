"""lrc_fro_diff_noalloc: the Frobenius reduction for callers that cannot
allocate device memory.

Who needs it: code that runs inside a fixed device-memory budget whose memory
belongs to another allocator (for example a serving framework's caching
pool), and latency-critical loops that cannot take the implicit device
synchronisation a cudaMalloc may cause.  The entry point keeps its per-block
partial sums in a fixed array inside the library instead of allocating.

These tests call it through the C ABI and compare it with lrc_fro_diff, the
allocating entry point, and with the oracle, at the 1e-12 relative tolerance
the other fro_diff tests use.  The file name makes pytest collect it last.
"""
import ctypes

import pytest
import torch

import oracle
import workloads as W
from parity import to_dev

pytestmark = pytest.mark.gpu

TOL = 1e-12
F64, F16 = 0, 2


def call(fn, A, fa, B, fb, count):
    diff = ctypes.c_double(-1.0)
    norm = ctypes.c_double(-1.0)
    status = fn(A.data_ptr(), fa, B.data_ptr() if B is not None else None, fb, count,
                ctypes.addressof(diff), ctypes.addressof(norm), torch.cuda.current_stream().cuda_stream)
    return status, diff.value, norm.value


def test_noalloc_agrees_with_lrc_fro_diff_on_two_calls_in_a_row(lrc, cuda):
    L = lrc.load()
    # call 1: a large FP64 pair; call 2: a smaller mixed FP64 / binary16 pair,
    # which uses fewer partial-sum slots than call 1 left behind
    a1 = W.gaussian((6_000_003,), 1)
    b1 = a1 + W.gaussian((6_000_003,), 2, 1e-3)
    a2 = W.gaussian((777_777,), 3)
    b2 = W.gaussian((777_777,), 4)
    A1, B1 = to_dev(a1, cuda), to_dev(b1, cuda)
    A2, B2 = to_dev(a2, cuda), to_dev(b2, cuda).half()
    ref1 = call(L.lrc_fro_diff, A1, F64, B1, F64, a1.size)
    ref2 = call(L.lrc_fro_diff, A2, F64, B2, F16, a2.size)
    got1 = call(L.lrc_fro_diff_noalloc, A1, F64, B1, F64, a1.size)
    got2 = call(L.lrc_fro_diff_noalloc, A2, F64, B2, F16, a2.size)
    want1 = oracle.fro_diff(a1, b1)
    want2 = oracle.fro_diff(a2, B2.double().cpu().numpy())
    for ref, got, want in ((ref1, got1, want1), (ref2, got2, want2)):
        assert ref[0] == 0 and got[0] == 0
        assert abs(got[1] - ref[1]) <= TOL * ref[1]
        assert abs(got[2] - ref[2]) <= TOL * ref[2]
        assert abs(got[1] - want[0]) <= TOL * want[0]
        assert abs(got[2] - want[1]) <= TOL * want[1]


def test_noalloc_without_the_norm(lrc, cuda):
    """normA_out = NULL: the difference alone, same value as with the norm."""
    L = lrc.load()
    a = W.gaussian((1_234_567,), 5)
    b = a + W.gaussian((1_234_567,), 6, 1e-6)
    A, B = to_dev(a, cuda), to_dev(b, cuda)
    with_norm = call(L.lrc_fro_diff_noalloc, A, F64, B, F64, a.size)
    diff = ctypes.c_double(-1.0)
    status = L.lrc_fro_diff_noalloc(A.data_ptr(), F64, B.data_ptr(), F64, a.size, ctypes.addressof(diff),
                                    None, torch.cuda.current_stream().cuda_stream)
    assert status == 0 and with_norm[0] == 0
    assert abs(diff.value - with_norm[1]) <= TOL * with_norm[1]
    want = oracle.fro_diff(a, b)[0]
    assert abs(diff.value - want) <= TOL * want


def test_noalloc_rejects_counts_beyond_its_fixed_array(lrc, cuda):
    L = lrc.load()
    diff = ctypes.c_double(0.0)
    status = L.lrc_fro_diff_noalloc(16, F64, None, F64, 268_435_456 + 1, ctypes.addressof(diff), None, None)
    assert status == -1
    assert b"at most 268435456" in L.lrc_last_error()
