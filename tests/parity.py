"""Shared helpers for the GPU parity tests: move seeded FP64 inputs to the
device, round them through the library, and compare with the oracle."""
import numpy as np

import oracle

# relative Frobenius tolerances per path
# bf16: 4 u with u = 2^-8, the multiple of the unit roundoff the FP16-output
# bar uses (2e-3 ~ 4 x 2^-11): W and the output are each rounded once to
# bfloat16, a relative Frobenius error of at most about 2u
TOL = {"f64": 1e-12, "f32": 1e-5, "f16": 1e-5, "f16_o16": 2e-3, "f32tc": 1e-5, "bf16": 4 * 2.0 ** -8}
BITS_DTYPE = {"f64": np.float64, "f32": np.uint32, "f16": np.uint16, "bf16": np.uint16}


def base_fmt(fmt: str) -> str:
    """Storage format whose rounding the oracle applies (f32tc stores binary32)."""
    return "f16" if fmt.startswith("f16") else ("f32" if fmt == "f32tc" else fmt)


def rel_fro(got: np.ndarray, want: np.ndarray) -> float:
    got = np.asarray(got, dtype=np.float64).reshape(-1)
    want = np.asarray(want, dtype=np.float64).reshape(-1)
    nw = float(np.linalg.norm(want))
    return float(np.linalg.norm(got - want)) / (nw if nw > 0 else 1.0)


def to_dev(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def packed(lrc, a64: np.ndarray, fmt: str, dev):
    """Round a host FP64 matrix through lrc_round_factors into a packed tensor."""
    a = a64 if a64.ndim == 2 else a64[None, :]
    return lrc.round_matrix(to_dev(a, dev), fmt)


def bits(t, fmt: str) -> np.ndarray:
    import torch
    if t.dtype == torch.bfloat16:            # numpy has no bfloat16: read the encodings
        t = t.view(torch.int16)
    return t.cpu().numpy().view(BITS_DTYPE[base_fmt(fmt)])


def host64(t) -> np.ndarray:
    """FP64 copy of a device tensor of any storage format (exact widening)."""
    return t.double().cpu().numpy()


def oracle_inputs(U, s, Vt, X, fmt):
    b = base_fmt(fmt)
    return (oracle.rounded(U, b), oracle.rounded(s, b), oracle.rounded(Vt, b), oracle.rounded(X, b))
