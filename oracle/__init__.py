"""CPU oracle for the rank-compensation hot path (FP64, plain C via ctypes).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline legs of ``bench.py`` may import this package.  The GPU
library (``paper_2607_12969_gb300``) never imports it, and the two share no
code: the only module both use is ``workloads`` (seeded inputs, no method
arithmetic).

Every function cites the passage of the paper it follows; the C source
(``oracle.c``) holds the arithmetic of the hot path.  The factorization side
(TT-SVD, left-orthogonalization) takes LAPACK's SVD and QR, through numpy, as
the primitive of each step of the paper's algorithm.  Inputs that the GPU sees in FP32/FP16
are given to the oracle as the oracle's own rounding of the FP64 data,
decoded back to FP64 exactly, so both sides evaluate the same rounded
factors.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
from typing import List, Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")

FMT_CODE = {"f64": 0, "f32": 1, "f16": 2, "bf16": 3}
BITS = {"f64": 64, "f32": 32, "f16": 16, "bf16": 16}
# unit roundoff u = 2^-p (Sec. 3.2, Table "precision comparison")
UNIT_ROUNDOFF = {"f64": 2.0 ** -53, "f32": 2.0 ** -24, "f16": 2.0 ** -11, "bf16": 2.0 ** -8}
ENC_DTYPE = {"f64": np.float64, "f32": np.uint32, "f16": np.uint16, "bf16": np.uint16}


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so with gcc (IEEE semantics kept:
    no fast-math, no FMA contraction)."""
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-ffp-contract=off", "-fno-fast-math",
           "-shared", "-fPIC", _SRC, "-o", _LIB + ".tmp", "-lm"]
    subprocess.check_call(cmd)
    os.replace(_LIB + ".tmp", _LIB)
    return _LIB


_lib = None


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        L = ctypes.CDLL(_LIB)
        i64, dbl, vp, ip = ctypes.c_int64, ctypes.c_double, ctypes.c_void_p, ctypes.c_int
        L.oracle_f64_to_f32_bits.restype = ctypes.c_uint32
        L.oracle_f64_to_f32_bits.argtypes = [dbl]
        L.oracle_f64_to_f16_bits.restype = ctypes.c_uint16
        L.oracle_f64_to_f16_bits.argtypes = [dbl]
        L.oracle_f64_to_bf16_bits.restype = ctypes.c_uint16
        L.oracle_f64_to_bf16_bits.argtypes = [dbl]
        L.oracle_round_pack.argtypes = [vp, i64, i64, i64, vp, i64, ip]
        L.oracle_decode.argtypes = [vp, i64, ip, vp]
        L.oracle_apply.argtypes = [vp, i64, vp, vp, i64, vp, i64, vp, i64, i64, i64, i64, i64]
        L.oracle_apply_rows.argtypes = [vp, i64, vp, vp, i64, vp, i64, vp, i64, vp, i64, i64, i64]
        L.oracle_tt_chain.argtypes = [vp, vp, vp, ip, vp]
        L.oracle_tt_chain.restype = ip
        L.oracle_tt_entries.argtypes = [vp, vp, vp, ip, vp, i64, vp]
        L.oracle_tt_entries.restype = ip
        L.oracle_fro_diff.argtypes = [vp, vp, i64, vp, vp]
        L.oracle_tail_error.argtypes = [vp, i64, i64]
        L.oracle_tail_error.restype = dbl
        L.oracle_certified.argtypes = [dbl, dbl, dbl]
        L.oracle_certified.restype = ip
        L.oracle_matrix_bound.argtypes = [dbl, dbl, dbl]
        L.oracle_matrix_bound.restype = dbl
        L.oracle_matrix_storage_bits.argtypes = [i64, i64, i64, ip]
        L.oracle_matrix_storage_bits.restype = dbl
        L.oracle_tt_storage_bits.argtypes = [vp, vp, ip, ip]
        L.oracle_tt_storage_bits.restype = dbl
        L.oracle_threads.restype = ip
        L.oracle_set_threads.argtypes = [ip]
        _lib = L
    return _lib


def _p(a: np.ndarray) -> int:
    return a.ctypes.data


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def threads() -> int:
    return int(lib().oracle_threads())


def set_threads(n: int) -> None:
    """Number of OpenMP threads the oracle's loops use (results unchanged)."""
    lib().oracle_set_threads(int(n))


# --------------------------------------------------------------------------
# rounding (Sec. 3.2-3.3; factors rounded individually, remark after Thm 4.1)
# --------------------------------------------------------------------------

def packed_ld(cols: int) -> int:
    """Row pitch of a packed factor: cols rounded up to a multiple of 16."""
    return ((int(cols) + 15) // 16) * 16


def round_pack(src: np.ndarray, fmt: str, ld: Optional[int] = None) -> np.ndarray:
    """RN-even rounding of a 2-D FP64 array to fmt, rows padded with +0 to ld.

    Returns the encodings: float64 for f64, uint32 for f32, uint16 for f16
    and bf16."""
    src = _f64(src)
    if src.ndim == 1:
        src = src[None, :]
    rows, cols = src.shape
    ld = cols if ld is None else ld
    out = np.empty((rows, ld), dtype=ENC_DTYPE[fmt])
    lib().oracle_round_pack(_p(src), rows, cols, cols, _p(out), ld, FMT_CODE[fmt])
    return out


def round_bits(x: np.ndarray, fmt: str) -> np.ndarray:
    """Element-wise RN-even encodings of an FP64 array (any shape)."""
    x = _f64(x)
    flat = x.reshape(1, -1) if x.size else x.reshape(1, 0)
    return round_pack(flat, fmt).reshape(x.shape)


def decode(bits: np.ndarray, fmt: str) -> np.ndarray:
    """Exact FP64 values of encodings produced by round_bits / the GPU."""
    b = np.ascontiguousarray(bits, dtype=ENC_DTYPE[fmt])
    out = np.empty(b.shape, dtype=np.float64)
    lib().oracle_decode(_p(b), b.size, FMT_CODE[fmt], _p(out))
    return out


def rounded(x: np.ndarray, fmt: str) -> np.ndarray:
    """FP64 value of x stored in fmt (round, then decode exactly)."""
    if fmt == "f64":
        return _f64(x).copy()
    return decode(round_bits(x, fmt), fmt)


# --------------------------------------------------------------------------
# matrix apply (Sec. 4.4, Eq. gpu_matrix_apply)
# --------------------------------------------------------------------------

def apply(U: np.ndarray, s: np.ndarray, Vt: np.ndarray, X: np.ndarray) -> np.ndarray:
    """Y = [(X V) diag(s)] U^T in FP64; U m x k, s k, Vt k x n, X b x n."""
    U, s, Vt, X = _f64(U), _f64(s), _f64(Vt), _f64(X)
    m, k = U.shape
    n = Vt.shape[1]
    b = X.shape[0]
    assert Vt.shape[0] == k and s.shape == (k,) and X.shape[1] == n
    Y = np.empty((b, m), dtype=np.float64)
    lib().oracle_apply(_p(U), k, _p(s), _p(Vt), n, _p(X), n, _p(Y), m, m, n, k, b)
    return Y


def apply_rows(U, s, Vt, X, rows: Sequence[int]) -> np.ndarray:
    """Rows `rows` of apply(U, s, Vt, X), without evaluating the others."""
    U, s, Vt, X = _f64(U), _f64(s), _f64(Vt), _f64(X)
    m, k = U.shape
    n = Vt.shape[1]
    r = np.ascontiguousarray(rows, dtype=np.int64)
    Y = np.empty((r.size, m), dtype=np.float64)
    lib().oracle_apply_rows(_p(U), k, _p(s), _p(Vt), n, _p(X), n, _p(r), r.size, _p(Y), m, n, k)
    return Y


# --------------------------------------------------------------------------
# TT reconstruction (Sec. 5.1 definition; Sec. 7.5 Eq. gpu_tt_reconstruction)
# --------------------------------------------------------------------------

def _tt_args(cores: Sequence[np.ndarray]):
    cs = [_f64(c) for c in cores]
    d = len(cs)
    dims = np.array([c.shape[1] for c in cs], dtype=np.int64)
    ranks = np.array([cs[0].shape[0]] + [c.shape[2] for c in cs], dtype=np.int64)
    for l in range(d - 1):
        assert cs[l].shape[2] == cs[l + 1].shape[0]
    ptrs = (ctypes.c_void_p * d)(*[c.ctypes.data for c in cs])
    return cs, d, dims, ranks, ptrs


def tt_full(cores: Sequence[np.ndarray]) -> np.ndarray:
    """Dense tensor by the reshape / product chain of Eq. gpu_tt_reconstruction."""
    cs, d, dims, ranks, ptrs = _tt_args(cores)
    out = np.empty(int(np.prod(dims)), dtype=np.float64)
    rc = lib().oracle_tt_chain(ptrs, _p(dims), _p(ranks), d, _p(out))
    if rc != 0:
        raise MemoryError(f"oracle_tt_chain failed ({rc})")
    return out.reshape(tuple(int(x) for x in dims))


def tt_entries(cores: Sequence[np.ndarray], flat_idx: Sequence[int]) -> np.ndarray:
    """Entries T(i_1..i_d) = G_1(i_1)...G_d(i_d) (Sec. 5.1) at C-order flat indices."""
    cs, d, dims, ranks, ptrs = _tt_args(cores)
    f = np.ascontiguousarray(flat_idx, dtype=np.int64)
    out = np.empty(f.size, dtype=np.float64)
    rc = lib().oracle_tt_entries(ptrs, _p(dims), _p(ranks), d, _p(f), f.size, _p(out))
    if rc != 0:
        raise MemoryError(f"oracle_tt_entries failed ({rc})")
    return out


# --------------------------------------------------------------------------
# Frobenius difference, eta and the certificates
# --------------------------------------------------------------------------

def fro_diff(a: np.ndarray, b: Optional[np.ndarray] = None) -> Tuple[float, float]:
    """(||a - b||_F, ||a||_F), Neumaier-compensated FP64 sums (Sec. 5.1)."""
    a = _f64(a).reshape(-1)
    bb = None if b is None else _f64(b).reshape(-1)
    if bb is not None:
        assert bb.size == a.size
    d = np.zeros(1)
    na = np.zeros(1)
    lib().oracle_fro_diff(_p(a), 0 if bb is None else _p(bb), a.size, _p(d), _p(na))
    return float(d[0]), float(na[0])


def eta_matrix(U, s, Vt, fmt: str) -> float:
    """eta = ||A_k' - Ahat_k'||_F (Thm 4.1 and the remark after it): U, s, Vt
    rounded individually to fmt, both products formed in FP64 (dense)."""
    n = Vt.shape[1]
    I = np.eye(n)
    A = apply(U, s, Vt, I)
    Ah = apply(rounded(U, fmt), rounded(s, fmt), rounded(Vt, fmt), I)
    return fro_diff(A, Ah)[0]


def eta_tt(cores: Sequence[np.ndarray], fmt: str) -> float:
    """eta_TT = ||T_R+ - That_R+||_F (Thm 6.1, Sec. 6.1): rounded cores
    reconstructed in FP64."""
    T = tt_full(cores)
    Th = tt_full([rounded(c, fmt) for c in cores])
    return fro_diff(T, Th)[0]


def tail_error(sigma: np.ndarray, k: int) -> float:
    """E_k = (sum_{j>k} sigma_j^2)^(1/2) (Sec. 4)."""
    sg = _f64(sigma)
    return float(lib().oracle_tail_error(_p(sg), sg.size, int(k)))


def certified(e_base: float, e_aug: float, eta: float) -> bool:
    """Eq. matrix_condition / Eq. tt_condition: E_aug + eta <= E_base."""
    return bool(lib().oracle_certified(float(e_base), float(e_aug), float(eta)))


def matrix_bound(e_k: float, sigma_next: float, eta: float) -> float:
    """Eq. matrix_universal_bound."""
    return float(lib().oracle_matrix_bound(float(e_k), float(sigma_next), float(eta)))


def matrix_storage_ratio(m: int, n: int, k_base: int, k_aug: int, fmt: str) -> float:
    """Eq. matrix_storage_ratio generalised to rank k_aug >= k_base."""
    L = lib()
    return (L.oracle_matrix_storage_bits(m, n, k_aug, BITS[fmt])
            / L.oracle_matrix_storage_bits(m, n, k_base, 64))


def tt_storage_bits(dims: Sequence[int], ranks: Sequence[int], fmt: str) -> float:
    dd = np.ascontiguousarray(dims, dtype=np.int64)
    rr = np.ascontiguousarray(ranks, dtype=np.int64)
    return float(lib().oracle_tt_storage_bits(_p(dd), _p(rr), dd.size, BITS[fmt]))


def tt_storage_ratio(dims, ranks_base, ranks_aug, fmt: str) -> float:
    """Exact TT storage ratio from the core dimensions (Sec. 6.1)."""
    return tt_storage_bits(dims, ranks_aug, fmt) / tt_storage_bits(dims, ranks_base, "f64")


# --------------------------------------------------------------------------
# factorization side: TT-SVD and left-orthogonalization (Sec. 5, Sec. 6.1)
# --------------------------------------------------------------------------

def tt_svd(T: np.ndarray, ranks: Sequence[int]):
    """TT-SVD (Sec. 5: the sequential truncated SVDs of Oseledets' algorithm;
    Alg. alg:tt_compensation steps 1-2).  The remainder C starts as T; at bond
    l it is reshaped to (r_{l-1} n_l) x (rest), its SVD U s V^T is truncated
    to r_l = min(ranks[l], len(s)) terms, core l is U[:, :r_l] and the next
    remainder is diag(s[:r_l]) V^T[:r_l].  The library SVD (LAPACK) is the
    step's primitive.  Returns (cores, delta2): delta2[l - 1] = sum of the
    discarded s_j^2 at bond l (summed from the smallest up).  The error of
    the result is ||T - T_R||_F^2 = sum(delta2) (the discarded parts of the
    successive steps are orthogonal)."""
    import math
    A = _f64(T)
    dims = A.shape
    d = len(dims)
    C = A.reshape(-1)
    rp = 1
    cores, delta2 = [], []
    for l in range(d - 1):
        C = C.reshape(rp * dims[l], -1)
        U, s, Vt = np.linalg.svd(C, full_matrices=False)
        r = min(int(ranks[l + 1]), s.size)
        delta2.append(math.fsum((s[r:] ** 2)[::-1]))
        cores.append(np.ascontiguousarray(U[:, :r].reshape(rp, dims[l], r)))
        C = s[:r, None] * Vt[:r]
        rp = r
    cores.append(np.ascontiguousarray(C.reshape(rp, dims[-1], 1)))
    return cores, delta2


def tt_left_orthogonalize(cores: Sequence[np.ndarray]):
    """Left-orthogonal gauge (Sec. 6.1): for l = 1..d-1 the unfolding
    (r_{l-1} n_l) x r_l of core l is factored Q R (LAPACK QR), core l becomes
    Q and R multiplies core l + 1 from the left.  The tensor is unchanged."""
    cs = [_f64(c).copy() for c in cores]
    for l in range(len(cs) - 1):
        r0, n, r1 = cs[l].shape
        Q, R = np.linalg.qr(cs[l].reshape(r0 * n, r1))
        k = Q.shape[1]
        cs[l] = np.ascontiguousarray(Q.reshape(r0, n, k))
        nxt = cs[l + 1]
        cs[l + 1] = np.ascontiguousarray((R @ nxt.reshape(nxt.shape[0], -1)).reshape(k, nxt.shape[1], nxt.shape[2]))
    return cs
