"""The C-ABI library loads, exports every symbol include/lrc.h declares, and
its host-only logic (validation that rejects before any launch, certificate
and storage helpers) behaves as specified -- all without a GPU."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import paper_2607_12969_gb300 as lrc
import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    if not os.path.exists(lrc.LIB_PATH):
        import __graft_entry__
        __graft_entry__.build()
    return lrc.load()


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "lrc.h")).read()
    return re.findall(r"LRC_API\s+[\w\s\*]+?\b(\w+)\s*\(", text)


def test_header_declares_the_boundary():
    names = set(declared_symbols())
    for required in ("lrc_round_factors", "lrc_apply", "tt_reconstruct", "lrc_fro_diff",
                     "lrc_widen_factors", "lrc_packed_ld", "lrc_certified"):
        assert required in names


def test_every_declared_symbol_is_exported(L):
    for name in declared_symbols():
        assert hasattr(L, name), name
        assert ctypes.cast(getattr(L, name), ctypes.c_void_p).value


def test_packed_ld(L):
    assert [lrc.lrc_packed_ld(c) for c in (0, 1, 15, 16, 17, 144, 8192)] == [0, 16, 16, 16, 32, 144, 8192]
    assert lrc.lrc_packed_ld(-1) == -1


def test_validation_rejects_before_launch(L):
    # null pointers / bad sizes / bad formats are rejected on the host
    st = L.lrc_apply(None, None, None, None, None, 4, 4, 2, 1, 0, None)
    assert st == -1
    st = L.lrc_apply(16, 16, 16, 16, 16, 0, 4, 2, 1, 0, None)
    assert st == -1
    st = L.lrc_apply(16, 16, 16, 16, 16, 4, 4, 2, 1, 7, None)
    assert st == -1
    st = L.lrc_apply(16, 16, 16, 16, 16, 4, 4, 2, 1, 6, None)       # one past LRC_BF16
    assert st == -1
    st = L.lrc_apply(17, 16, 16, 16, 16, 4, 4, 2, 1, 5, None)       # LRC_BF16 is a format: checks go on
    assert st == -2
    st = L.lrc_apply(17, 16, 16, 16, 16, 4, 4, 2, 1, 4, None)       # LRC_F32_TC is a format: checks go on
    assert st == -2
    st = L.lrc_apply(17, 16, 16, 16, 16, 4, 4, 2, 1, 0, None)      # misaligned U
    assert st == -2
    st = L.lrc_round_factors(16, 4, 8, 4, 16, 8, 1, None)           # ld_src < cols
    assert st == -1
    st = L.lrc_round_factors(16, 0, 8, 8, 16, 8, 1, None)           # nothing to do
    assert st == 0
    st = L.lrc_round_factors(16, 4, 8, 8, 24, 8, 2, None)           # misaligned dst
    assert st == -2
    d = ctypes.c_double(-1.0)
    assert L.lrc_fro_diff(None, 0, None, 0, 0, ctypes.addressof(d), None, None) == 0 and d.value == 0.0
    assert L.lrc_fro_diff(None, 0, None, 0, -1, ctypes.addressof(d), None, None) == -1
    assert "count" in L.lrc_last_error().decode()


def test_tt_validation(L):
    dims = (ctypes.c_int64 * 3)(4, 5, 6)
    ranks_bad = (ctypes.c_int64 * 4)(2, 3, 3, 1)
    ptrs = (ctypes.c_void_p * 3)(16, 16, 16)
    st = L.tt_reconstruct(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dims, ctypes.c_void_p),
                          ctypes.cast(ranks_bad, ctypes.c_void_p), 3, 0, 16, None)
    assert st == -1
    ranks = (ctypes.c_int64 * 4)(1, 3, 3, 1)
    st = L.tt_reconstruct(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dims, ctypes.c_void_p),
                          ctypes.cast(ranks, ctypes.c_void_p), 1, 0, 16, None)
    assert st == -1
    st = L.tt_reconstruct(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dims, ctypes.c_void_p),
                          ctypes.cast(ranks, ctypes.c_void_p), 3, 0, 8, None)   # misaligned out
    assert st == -2
    zero = (ctypes.c_int64 * 3)(4, 0, 6)
    st = L.tt_reconstruct(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(zero, ctypes.c_void_p),
                          ctypes.cast(ranks, ctypes.c_void_p), 3, 0, 16, None)
    assert st == -1


def test_host_helpers_agree_with_oracle(L):
    rng = np.random.default_rng(0)
    for _ in range(500):
        eb, ea, eta = rng.uniform(0, 1, 3)
        assert lrc.lrc_certified(eb, ea, eta) == oracle.certified(eb, ea, eta)
    sig = W.spectrum("alg1.5", 1000)
    for k in (0, 1, 128, 136, 999, 1000):
        assert lrc.lrc_tail_error(sig, k) == oracle.tail_error(sig, k)
    for fmt in ("f32", "f16"):
        assert abs(lrc.lrc_matrix_storage_ratio(16384, 8192, 128, 144, fmt)
                   - oracle.matrix_storage_ratio(16384, 8192, 128, 144, fmt)) < 1e-15
        dims, base, aug = (256, 256, 256), (1, 32, 32, 1), (1, 34, 34, 1)
        assert abs(lrc.lrc_tt_storage_bytes(dims, aug, fmt) * 8 - oracle.tt_storage_bits(dims, aug, fmt)) < 1e-6
    assert lrc.lrc_matrix_storage_ratio(10, 10, 40, 41, "f16") == pytest.approx(0.25625)
    # the binary32 tensor-core variant stores binary32
    assert lrc.lrc_matrix_storage_ratio(16384, 8192, 128, 136, "f32tc") == \
        lrc.lrc_matrix_storage_ratio(16384, 8192, 128, 136, "f32")


def test_eta_validation_rejects_before_launch(L):
    """lrc_lowrank_eta / lrc_tt_eta reject bad arguments on the host."""
    out = ctypes.c_double(0.0)
    po = ctypes.addressof(out)
    # null factor, zero size, bad format, misaligned pointer, k too large
    assert L.lrc_lowrank_eta(None, 16, 16, 16, 16, 16, 2, 4, 4, 2, po, None, None) == -1
    assert L.lrc_lowrank_eta(16, 16, 16, 16, 16, 16, 2, 0, 4, 2, po, None, None) == -1
    assert L.lrc_lowrank_eta(16, 16, 16, 16, 16, 16, 9, 4, 4, 2, po, None, None) == -1
    assert L.lrc_lowrank_eta(16, 16, 16, 24, 16, 16, 2, 4, 4, 2, po, None, None) == -2
    assert L.lrc_lowrank_eta(16, 16, 16, 16, 16, 16, 2, 4, 4, 5000, po, None, None) == -1
    assert L.lrc_lowrank_eta(16, 16, 16, 16, 16, 16, 2, 4, 4, 2, None, None, None) == -1
    d = 3
    c = (ctypes.c_void_p * d)(16, 16, 16)
    ch = (ctypes.c_void_p * d)(16, 16, 16)
    dims = (ctypes.c_int64 * d)(4, 5, 6)
    bad = (ctypes.c_int64 * (d + 1))(2, 3, 3, 1)          # r_0 != 1
    assert L.lrc_tt_eta(c, ch, dims, bad, d, 2, po, None, None) == -1
    good = (ctypes.c_int64 * (d + 1))(1, 3, 3, 1)
    assert L.lrc_tt_eta(c, ch, dims, good, 1, 2, po, None, None) == -1   # d < 2
    assert L.lrc_tt_eta(c, ch, dims, good, d, 2, None, None, None) == -1  # null eta_out
    nul = (ctypes.c_void_p * d)(16, None, 16)
    assert L.lrc_tt_eta(c, nul, dims, good, d, 2, po, None, None) == -1
    odd = (ctypes.c_void_p * d)(16, 20, 16)                 # binary64 core not 8-byte aligned
    assert L.lrc_tt_eta(odd, ch, dims, good, d, 0, po, None, None) == -2


def test_gather_validation_rejects_before_launch(L):
    d = 2
    c = (ctypes.c_void_p * d)(16, 16)
    dims = (ctypes.c_int64 * d)(4, 5)
    ranks = (ctypes.c_int64 * (d + 1))(1, 3, 1)
    assert L.tt_gather(c, dims, ranks, d, 0, 16, -1, 16, None) == -1            # negative count
    assert L.tt_gather(c, dims, ranks, d, 0, 16, 0, 16, None) == 0              # nothing to do
    assert L.tt_gather(c, dims, ranks, d, 0, None, 3, 16, None) == -1           # null idx
    assert L.tt_gather(c, dims, ranks, d, 0, 12, 3, 16, None) == -2             # idx misaligned
    assert L.tt_gather(c, dims, ranks, d, 0, 16, 3, 20, None) == -2             # out misaligned (f64)
    big = (ctypes.c_int64 * (d + 1))(1, 300, 1)
    assert L.tt_gather(c, dims, big, d, 0, 16, 3, 16, None) == -3               # rank above 256
