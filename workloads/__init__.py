"""Seeded synthetic inputs for the rank-compensation hot path.

This module is shared by the CPU oracle (``oracle/``) and by the GPU path's
tests and benchmark.  It holds no arithmetic of the method itself (no
rounding, no apply, no contraction, no norm): it only draws seeded FP64 data
with the shapes, spectra and structure of the paper's workloads.

* Matrix factors follow the truncated-SVD model of Sec. 4: ``A = Q1 diag(sigma)
  Q2^T`` with ``Q1``, ``Q2`` from the QR factorisation of seeded N(0,1)
  matrices, diagonal of R made positive.  Factors are nested: the rank-k
  factors are the leading k columns of the same ``Q1``/``Q2`` used for rank
  k' > k, as for a truncated SVD.
* The query batch ``X`` (b x n, one query per row) is seeded N(0,1)
  (Sec. 4.4 draws standard-normal queries).
* TT cores follow Sec. 5.1 (cores ``R_{l-1} x n_l x R_l``, ``R_0 = R_d = 1``)
  in the left-orthogonal gauge of Sec. 6.1: cores 1..d-1 have orthonormal
  columns when reshaped to ``(R_{l-1} n_l) x R_l`` and the last core is
  ``diag(lambda) W`` with ``W`` having orthonormal rows, so that
  ``||T||_F = ||lambda||_2`` exactly.  Ranks are capped by the valid unfolding
  dimension as in Sec. 7.4.

Seeds are ``1000*cfg + stream``: stream 1 = Q1, 2 = Q2, 3 = X, 10+l = TT core
l; +100 for the FP32 rank set and +200 for the FP16 rank set of a TT config.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, List, Sequence, Tuple

import numpy as np

FORMATS = ("f64", "f32", "f16")


# ---------------------------------------------------------------------------
# configurations (the five synthetic workloads)
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class MatrixConfig:
    name: str
    cfg: int
    m: int
    n: int
    b: int
    ranks: Dict[str, int]          # format -> rank (f64 = base rank k)
    spectrum: str                  # "pow2_16" (sigma_j = 2^(-j/16)) or "alg1.5" (j^-1.5)

    @property
    def k_max(self) -> int:
        return max(self.ranks.values())


@dataclasses.dataclass(frozen=True)
class TTConfig:
    name: str
    cfg: int
    dims: Tuple[int, ...]
    ranks: Dict[str, Tuple[int, ...]]   # format -> full rank vector (1, R_1, ..., 1)
    kind: str                           # "gauss_geo", "gauss_alg", "smooth"


def capped_ranks(dims: Sequence[int], r: int) -> Tuple[int, ...]:
    """Uniform nominal rank capped by the unfolding dimension (Sec. 7.4)."""
    d = len(dims)
    out = [1]
    for l in range(1, d):
        left = int(np.prod(dims[:l]))
        right = int(np.prod(dims[l:]))
        out.append(min(r, left, right))
    out.append(1)
    return tuple(out)


MATRIX_CONFIGS: Dict[str, MatrixConfig] = {
    "tiny": MatrixConfig("tiny", 1, 512, 512, 64, {"f64": 32, "f32": 33, "f16": 34}, "pow2_16"),
    "large": MatrixConfig("large", 2, 16384, 8192, 8192, {"f64": 128, "f32": 136, "f16": 144}, "alg1.5"),
}

SWEEP_BATCHES = (1, 16, 256, 4096, 32768)


def sweep_config(b: int) -> MatrixConfig:
    """Apply batch sweep of the hyperspectral-shaped workload (m = n = 16384)."""
    return MatrixConfig(f"sweep_b{b}", 5, 16384, 16384, b,
                        {"f64": 256, "f32": 272, "f16": 272}, "alg1.5")


TT_CONFIGS: Dict[str, TTConfig] = {
    "tt3": TTConfig("tt3", 3, (256, 256, 256),
                    {"f64": (1, 32, 32, 1), "f32": (1, 34, 34, 1), "f16": (1, 34, 34, 1)},
                    "gauss_geo"),
    "tt6": TTConfig("tt6", 4, (16,) * 6,
                    {"f64": capped_ranks((16,) * 6, 24), "f32": capped_ranks((16,) * 6, 26),
                     "f16": capped_ranks((16,) * 6, 28)},
                    "gauss_alg"),
    "tt_hsi": TTConfig("tt_hsi", 5, (512, 512, 224),
                       {"f64": (1, 64, 48, 1), "f32": (1, 70, 52, 1), "f16": (1, 70, 52, 1)},
                       "smooth"),
}


# ---------------------------------------------------------------------------
# matrix factors and queries
# ---------------------------------------------------------------------------

def spectrum(kind: str, count: int) -> np.ndarray:
    """Singular values sigma_1 >= sigma_2 >= ... (1-based j)."""
    j = np.arange(1, count + 1, dtype=np.float64)
    if kind == "pow2_16":
        return np.exp2(-j / 16.0)
    if kind == "alg1.5":
        return j ** -1.5
    raise ValueError(kind)


def orthonormal_columns(rows: int, cols: int, seed: int) -> np.ndarray:
    """Q of a seeded Gaussian rows x cols matrix, diag(R) > 0 (LAPACK QR)."""
    rng = np.random.default_rng(seed)
    g = rng.standard_normal((rows, cols))
    q, r = np.linalg.qr(g)
    sgn = np.sign(np.diag(r))
    sgn[sgn == 0] = 1.0
    return np.ascontiguousarray(q * sgn)


@dataclasses.dataclass
class Factors:
    """FP64 rank-k factors: U (m x k), s (k), Vt (k x n), all C order."""
    U: np.ndarray
    s: np.ndarray
    Vt: np.ndarray

    @property
    def k(self) -> int:
        return self.s.shape[0]


def matrix_bases(cfg: MatrixConfig, k_max: int | None = None):
    """Q1 (m x K), sigma (min(m,n)), Q2 (n x K) with K = k_max."""
    K = cfg.k_max if k_max is None else k_max
    q1 = orthonormal_columns(cfg.m, K, 1000 * cfg.cfg + 1)
    q2 = orthonormal_columns(cfg.n, K, 1000 * cfg.cfg + 2)
    sig = spectrum(cfg.spectrum, min(cfg.m, cfg.n))
    return q1, sig, q2


def truncate(q1: np.ndarray, sig: np.ndarray, q2: np.ndarray, k: int) -> Factors:
    return Factors(np.ascontiguousarray(q1[:, :k]), np.ascontiguousarray(sig[:k]),
                   np.ascontiguousarray(q2[:, :k].T))


def matrix_factors(cfg: MatrixConfig, fmt: str) -> Factors:
    q1, sig, q2 = matrix_bases(cfg)
    return truncate(q1, sig, q2, cfg.ranks[fmt])


def queries(cfg: MatrixConfig, b: int | None = None, replica: int = 0) -> np.ndarray:
    """Seeded N(0,1) query batch X, b x n, one query per row.  `replica` r > 0
    draws an independent batch of the same shape (one per GPU when the
    benchmark runs replicas: weak scaling)."""
    rng = np.random.default_rng(1000 * cfg.cfg + 3 + 100000 * replica)
    bb = cfg.b if b is None else b
    return rng.standard_normal((bb, cfg.n))


def random_factors(m: int, n: int, k: int, seed: int, spec: str = "alg1.5") -> Factors:
    """Small seeded factor set for edge-case tests (any m, n, k)."""
    kk = min(k, m, n)
    q1 = orthonormal_columns(m, kk, seed)
    q2 = orthonormal_columns(n, kk, seed + 1)
    sig = spectrum(spec, k)
    U = np.zeros((m, k))
    Vt = np.zeros((k, n))
    U[:, :kk] = q1
    Vt[:kk, :] = q2.T
    if kk < k:  # rank beyond min(m, n): fill with seeded Gaussian columns
        rng = np.random.default_rng(seed + 2)
        U[:, kk:] = rng.standard_normal((m, k - kk)) / np.sqrt(m)
        Vt[kk:, :] = rng.standard_normal((k - kk, n)) / np.sqrt(n)
    return Factors(U, sig, Vt)


def gaussian(shape, seed: int, scale: float = 1.0) -> np.ndarray:
    return np.random.default_rng(seed).standard_normal(shape) * scale


def integer_valued(shape, seed: int, lo: int = -8, hi: int = 8) -> np.ndarray:
    """Small integers as FP64: products and sums stay exact in every format."""
    return np.random.default_rng(seed).integers(lo, hi + 1, size=shape).astype(np.float64)


# ---------------------------------------------------------------------------
# TT cores
# ---------------------------------------------------------------------------

def _left_orthonormal_core(r0: int, n: int, r1: int, rng, row_scale=None) -> np.ndarray:
    g = rng.standard_normal((r0 * n, r1))
    if row_scale is not None:
        g = g * np.repeat(row_scale, n)[:, None]
    q, r = np.linalg.qr(g)
    sgn = np.sign(np.diag(r))
    sgn[sgn == 0] = 1.0
    return np.ascontiguousarray((q * sgn).reshape(r0, n, r1))


def _last_core(r0: int, n: int, lam: np.ndarray, rng) -> np.ndarray:
    g = rng.standard_normal((n, r0))
    q, r = np.linalg.qr(g)           # n x r0, orthonormal columns
    sgn = np.sign(np.diag(r))
    sgn[sgn == 0] = 1.0
    w = (q * sgn).T                  # r0 x n, orthonormal rows
    return np.ascontiguousarray((lam[:, None] * w).reshape(r0, n, 1))


def tt_last_spectrum(kind: str, r: int) -> np.ndarray:
    j = np.arange(1, r + 1, dtype=np.float64)
    if kind == "gauss_geo":
        return 0.9 ** j
    return 1.0 / j


def tt_cores(cfg: TTConfig, fmt: str) -> List[np.ndarray]:
    """Seeded FP64 cores for one rank set of a TT config (C order, r0 x n x r1)."""
    dims = cfg.dims
    ranks = cfg.ranks[fmt]
    off = {"f64": 0, "f32": 100, "f16": 200}[fmt]
    return make_tt(dims, ranks, cfg.kind, seed_base=1000 * cfg.cfg + off)


def make_tt(dims: Sequence[int], ranks: Sequence[int], kind: str, seed_base: int) -> List[np.ndarray]:
    d = len(dims)
    assert len(ranks) == d + 1 and ranks[0] == 1 and ranks[-1] == 1
    cores: List[np.ndarray] = []
    if kind in ("gauss_geo", "gauss_alg"):
        for l in range(d - 1):
            rng = np.random.default_rng(seed_base + 10 + l + 1)
            rs = None
            if kind == "gauss_alg":
                rs = 1.0 / np.arange(1, ranks[l] + 1, dtype=np.float64)
            cores.append(_left_orthonormal_core(ranks[l], dims[l], ranks[l + 1], rng, rs))
        rng = np.random.default_rng(seed_base + 10 + d)
        cores.append(_last_core(ranks[d - 1], dims[d - 1], tt_last_spectrum(kind, ranks[d - 1]), rng))
        return cores
    if kind == "smooth":
        raw = []
        for l in range(d):
            rng = np.random.default_rng(seed_base + 10 + l + 1)
            nq = 8
            c = rng.standard_normal((ranks[l], nq, ranks[l + 1]))
            i = np.arange(dims[l], dtype=np.float64)
            q = np.arange(nq, dtype=np.float64)
            basis = (1.0 + q)[:, None] ** -2 * np.cos(np.pi * q[:, None] * (i[None, :] + 0.5) / dims[l])
            raw.append(np.einsum("aqb,qi->aib", c, basis))
        # left-orthogonalisation sweep (QR, pass R to the right)
        for l in range(d - 1):
            r0, n, r1 = raw[l].shape
            q, r = np.linalg.qr(raw[l].reshape(r0 * n, r1))
            sgn = np.sign(np.diag(r))
            sgn[sgn == 0] = 1.0
            q = q * sgn
            r = sgn[:, None] * r
            raw[l] = np.ascontiguousarray(q.reshape(r0, n, r1))
            nxt = raw[l + 1]
            raw[l + 1] = np.einsum("ab,bic->aic", r, nxt)
        rng = np.random.default_rng(seed_base + 10 + d + 50)
        raw[d - 1] = _last_core(ranks[d - 1], dims[d - 1],
                                tt_last_spectrum("smooth", ranks[d - 1]), rng)
        return raw
    if kind == "gauss":
        out = []
        for l in range(d):
            rng = np.random.default_rng(seed_base + 10 + l + 1)
            out.append(rng.standard_normal((ranks[l], dims[l], ranks[l + 1])))
        return out
    raise ValueError(kind)


def tt_numel(dims: Sequence[int]) -> int:
    return int(np.prod(dims, dtype=np.int64))


def sample_indices(count: int, total: int, seed: int) -> np.ndarray:
    """Seeded distinct sample of flat indices in [0, total)."""
    rng = np.random.default_rng(seed)
    if count >= total:
        return np.arange(total, dtype=np.int64)
    return np.sort(rng.choice(total, size=count, replace=False)).astype(np.int64)


# ---------------------------------------------------------------------------
# the paper's closed-form three-way tensors (Sec. 7.2), C order, 1-based i, j, k
# ---------------------------------------------------------------------------

def hilbert_3d(n: int = 100) -> np.ndarray:
    """T(i, j, k) = 1 / (i + j + k - 2)."""
    i = np.arange(1, n + 1, dtype=np.float64)
    return 1.0 / (i[:, None, None] + i[None, :, None] + i[None, None, :] - 2.0)


def decay_3d(n: int = 60) -> np.ndarray:
    """T(i, j, k) = 1 / (1 + |i - j| + |j - k| + |i - k|)."""
    i = np.arange(1, n + 1, dtype=np.float64)
    a, b, c = i[:, None, None], i[None, :, None], i[None, None, :]
    return 1.0 / (1.0 + np.abs(a - b) + np.abs(b - c) + np.abs(a - c))
