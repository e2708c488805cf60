"""Python binding of liblrc.so, the GB300 rank-compensation hot path.

Argument marshalling only: every entry point forwards device pointers of
torch tensors (torch is used for device memory and streams) and sizes to the
C ABI declared in include/lrc.h, where every step runs in the library's own
CUDA kernels.  Before forwarding, it refuses tensors that are not CUDA
tensors of the format's element type, on the GPU the call runs on, with
storage for the extent the call reads or writes (the C ABI cannot see buffer
sizes or devices).  There is no CPU fallback: if the library is missing or
fails to load, every call raises.

Names follow the C ABI: lrc_round_factors, lrc_widen_factors, lrc_apply,
tt_reconstruct, lrc_fro_diff, plus the host helpers lrc_certified,
lrc_tail_error, lrc_matrix_storage_ratio and lrc_tt_storage_bytes.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence, Tuple

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "liblrc.so")

F64, F32, F16, F16_O16, F32_TC, BF16 = 0, 1, 2, 3, 4, 5
FORMATS = {"f64": F64, "f32": F32, "f16": F16, "f16_o16": F16_O16, "f32tc": F32_TC, "bf16": BF16}
STATUS = {0: "ok", -1: "invalid argument", -2: "misaligned pointer", -3: "unsupported",
          -4: "CUDA error", -5: "out of memory", -6: "device wait timed out"}


class LrcError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


_lib: Optional[ctypes.CDLL] = None


def load() -> ctypes.CDLL:
    """Load liblrc.so (built by build.py); raises if it is absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                           "`python -c 'import __graft_entry__ as g; g.build()'`")
    L = ctypes.CDLL(LIB_PATH)
    i64, i32, vp, dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p, ctypes.c_double
    L.lrc_packed_ld.argtypes = [i64]
    L.lrc_packed_ld.restype = i64
    L.lrc_round_factors.argtypes = [vp, i64, i64, i64, vp, i64, i32, vp]
    L.lrc_round_factors.restype = i32
    L.lrc_widen_factors.argtypes = [vp, i32, i64, i64, i64, vp, i64, vp]
    L.lrc_widen_factors.restype = i32
    L.lrc_apply.argtypes = [vp, vp, vp, vp, vp, i64, i64, i64, i64, i32, vp]
    L.lrc_apply.restype = i32
    L.lrc_apply_batched.argtypes = [i32, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32, vp]
    L.lrc_apply_batched.restype = i32
    L.tt_reconstruct.argtypes = [vp, vp, vp, i32, i32, vp, vp]
    L.tt_reconstruct.restype = i32
    L.lrc_fro_diff.argtypes = [vp, i32, vp, i32, i64, vp, vp, vp]
    L.lrc_fro_diff.restype = i32
    L.lrc_fro_diff_noalloc.argtypes = [vp, i32, vp, i32, i64, vp, vp, vp]
    L.lrc_fro_diff_noalloc.restype = i32
    L.tt_gather.argtypes = [vp, vp, vp, i32, i32, vp, i64, vp, vp]
    L.tt_gather.restype = i32
    L.lrc_lowrank_eta.argtypes = [vp, vp, vp, vp, vp, vp, i32, i64, i64, i64, vp, vp, vp]
    L.lrc_lowrank_eta.restype = i32
    L.lrc_tt_eta.argtypes = [vp, vp, vp, vp, i32, i32, vp, vp, vp]
    L.lrc_tt_eta.restype = i32
    L.lrc_certified.argtypes = [dbl, dbl, dbl]
    L.lrc_certified.restype = i32
    L.lrc_tail_error.argtypes = [vp, i64, i64]
    L.lrc_tail_error.restype = dbl
    L.lrc_matrix_storage_ratio.argtypes = [i64, i64, i64, i64, i32]
    L.lrc_matrix_storage_ratio.restype = dbl
    L.lrc_tt_storage_bytes.argtypes = [vp, vp, i32, i32]
    L.lrc_tt_storage_bytes.restype = dbl
    L.lrc_status_string.argtypes = [i32]
    L.lrc_status_string.restype = ctypes.c_char_p
    L.lrc_last_error.restype = ctypes.c_char_p
    L.lrc_launch_count.restype = ctypes.c_uint64
    L.lrc_shutdown.restype = i32
    L.lrc_device_status.argtypes = [vp]
    L.lrc_device_status.restype = i32
    L.lrc_tt_svd.argtypes = [vp, vp, vp, i32, vp, vp, vp, vp]
    L.lrc_tt_svd.restype = i32
    L.lrc_tt_left_orthogonalize.argtypes = [vp, vp, vp, i32, vp]
    L.lrc_tt_left_orthogonalize.restype = i32
    L.lrc_probe_peak.argtypes = [i32, i64, vp, vp]
    L.lrc_probe_peak.restype = i32
    L.lrc_selftest_wait_timeout.argtypes = [i64, vp]
    L.lrc_selftest_wait_timeout.restype = i32
    _lib = L
    return L


def _fmt(fmt) -> int:
    if isinstance(fmt, str):
        return FORMATS[fmt]
    return int(fmt)


def storage_dtype(fmt):
    import torch
    f = _fmt(fmt)
    return {F64: torch.float64, F32: torch.float32, F16: torch.float16, F16_O16: torch.float16,
            F32_TC: torch.float32, BF16: torch.bfloat16}[f]


def output_dtype(fmt):
    import torch
    f = _fmt(fmt)
    return {F64: torch.float64, F32: torch.float32, F16: torch.float32, F16_O16: torch.float16,
            F32_TC: torch.float32, BF16: torch.bfloat16}[f]


def _check(status: int) -> None:
    if status != 0:
        msg = load().lrc_last_error().decode(errors="replace")
        raise LrcError(status, msg)


def np_prod(xs) -> int:
    p = 1
    for x in xs:
        p *= int(x)
    return p


def _stream(stream) -> int:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _ptr(t) -> int:
    return 0 if t is None else t.data_ptr()


def _span(t) -> int:
    """Elements of t's storage from its first element on (views included)."""
    return t.untyped_storage().nbytes() // t.element_size() - t.storage_offset()


def _call_device(stream) -> int:
    """Ordinal of the GPU a call runs on: the stream's device when a torch
    stream is given, else the current device (whose stream a raw handle or
    None names)."""
    dev = getattr(stream, "device", None)
    if dev is not None:
        return dev.index if hasattr(dev, "index") else int(dev)
    import torch
    return torch.cuda.current_device()


def _need(t, what: str, dtype=None, elems: int = 0, stream=None) -> None:
    """Marshalling checks that keep a call from reaching memory it does not
    own: a CUDA tensor of the format's element type, on the GPU the call runs
    on, whose storage holds at least `elems` elements from its first one.
    (Layout and values are the library's to check; sizes <= 0 are left to its
    validation.)"""
    if t is None:
        raise ValueError(f"{what}: a tensor is required")
    if not t.is_cuda:
        raise ValueError(f"{what}: must be a CUDA tensor (got device {t.device})")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{what}: element type {t.dtype}, the format needs {dtype}")
    want = _call_device(stream)
    if t.device.index is not None and t.device.index != want:
        raise ValueError(f"{what}: on {t.device}, but the call runs on cuda:{want} (a kernel there "
                         "cannot address another GPU's memory)")
    if elems > 0 and _span(t) < elems:
        raise ValueError(f"{what}: storage holds {_span(t)} elements from its start, the call reads or "
                         f"writes {elems}")


def _extent(rows: int, cols: int, ld: int) -> int:
    """Elements a rows x cols array with row pitch ld spans."""
    return (rows - 1) * ld + cols if rows > 0 and cols > 0 else 0


# --------------------------------------------------------------------------
# entry points (same names and argument order as include/lrc.h)
# --------------------------------------------------------------------------

def lrc_packed_ld(cols: int) -> int:
    return int(load().lrc_packed_ld(int(cols)))


def lrc_round_factors(src, rows: int, cols: int, ld_src: int, dst, ld_dst: int, fmt, stream=None):
    import torch
    _need(src, "src", torch.float64, _extent(rows, cols, ld_src), stream=stream)
    _need(dst, "dst", storage_dtype(fmt), _extent(rows, ld_dst, ld_dst), stream=stream)
    _check(load().lrc_round_factors(_ptr(src), rows, cols, ld_src, _ptr(dst), ld_dst, _fmt(fmt),
                                    _stream(stream)))


def lrc_widen_factors(src, fmt, rows: int, cols: int, ld_src: int, dst, ld_dst: int, stream=None):
    import torch
    _need(src, "src", storage_dtype(fmt), _extent(rows, cols, ld_src), stream=stream)
    _need(dst, "dst", torch.float64, _extent(rows, ld_dst, ld_dst), stream=stream)
    _check(load().lrc_widen_factors(_ptr(src), _fmt(fmt), rows, cols, ld_src, _ptr(dst), ld_dst,
                                    _stream(stream)))


def lrc_apply(U, S, Vt, X, Y, m: int, n: int, k: int, b: int, fmt, stream=None):
    if m > 0 and n > 0 and k > 0 and b > 0:
        st, ldk, ldn = storage_dtype(fmt), lrc_packed_ld(k), lrc_packed_ld(n)
        _need(U, "U", st, _extent(m, k, ldk), stream=stream)
        _need(S, "S", st, k, stream=stream)
        _need(Vt, "Vt", st, _extent(k, n, ldn), stream=stream)
        _need(X, "X", st, _extent(b, n, ldn), stream=stream)
        _need(Y, "Y", output_dtype(fmt), b * m, stream=stream)
    _check(load().lrc_apply(_ptr(U), _ptr(S), _ptr(Vt), _ptr(X), _ptr(Y), m, n, k, b, _fmt(fmt),
                            _stream(stream)))


def lrc_apply_batched(U: Sequence, S: Sequence, Vt: Sequence, X: Sequence, Y: Sequence, m: Sequence[int],
                      n: Sequence[int], k: Sequence[int], b: Sequence[int], fmt, stream=None):
    """Several independent applies in one call: problem p is
    lrc_apply(U[p], S[p], Vt[p], X[p], Y[p], m[p], n[p], k[p], b[p], fmt)."""
    count = len(U)
    if not all(len(a) == count for a in (S, Vt, X, Y, m, n, k, b)):
        raise ValueError("every argument needs one entry per problem")
    st, ot = storage_dtype(fmt), output_dtype(fmt)
    for p in range(count):
        mp, np_, kp, bp = int(m[p]), int(n[p]), int(k[p]), int(b[p])
        if mp > 0 and np_ > 0 and kp > 0 and bp > 0:
            ldk, ldn = lrc_packed_ld(kp), lrc_packed_ld(np_)
            _need(U[p], f"U[{p}]", st, _extent(mp, kp, ldk), stream=stream)
            _need(S[p], f"S[{p}]", st, kp, stream=stream)
            _need(Vt[p], f"Vt[{p}]", st, _extent(kp, np_, ldn), stream=stream)
            _need(X[p], f"X[{p}]", st, _extent(bp, np_, ldn), stream=stream)
            _need(Y[p], f"Y[{p}]", ot, bp * mp, stream=stream)
    arr = lambda ts: (ctypes.c_void_p * max(count, 1))(*[_ptr(t) for t in ts])  # noqa: E731
    i64s = lambda xs: (ctypes.c_int64 * max(count, 1))(*[int(x) for x in xs])   # noqa: E731
    pu, ps, pv, px, py = arr(U), arr(S), arr(Vt), arr(X), arr(Y)
    am, an, ak, ab = i64s(m), i64s(n), i64s(k), i64s(b)
    c = lambda a: ctypes.cast(a, ctypes.c_void_p)   # noqa: E731
    _check(load().lrc_apply_batched(count, c(pu), c(ps), c(pv), c(px), c(py), c(am), c(an), c(ak), c(ab),
                                    _fmt(fmt), _stream(stream)))


def _need_cores(cores, dims, ranks, fmt, stream=None) -> bool:
    """Checks the cores; True when dims and ranks describe them (else the
    library's validation reports the mismatch)."""
    d = len(cores)
    shaped = len(dims) == d and len(ranks) == d + 1 and all(int(x) > 0 for x in list(dims) + list(ranks))
    for l, c in enumerate(cores):
        _need(c, f"cores[{l}]", storage_dtype(fmt),
              int(ranks[l]) * int(dims[l]) * int(ranks[l + 1]) if shaped else 0, stream=stream)
    return shaped


def tt_reconstruct(cores: Sequence, dims: Sequence[int], ranks: Sequence[int], fmt, out, stream=None):
    if _need_cores(cores, dims, ranks, fmt, stream):
        _need(out, "out", output_dtype(fmt), int(np_prod(dims)), stream=stream)
    d = len(cores)
    ptrs = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores])
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    _check(load().tt_reconstruct(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dd, ctypes.c_void_p),
                                 ctypes.cast(rr, ctypes.c_void_p), d, _fmt(fmt), _ptr(out),
                                 _stream(stream)))


def tt_gather(cores: Sequence, dims: Sequence[int], ranks: Sequence[int], fmt, idx, out, stream=None):
    """Entries of the TT at the flat indices `idx` (int64 CUDA tensor) into `out`."""
    import torch
    _need_cores(cores, dims, ranks, fmt, stream)
    _need(idx, "idx", torch.int64, stream=stream)
    gather_dtype = {F64: torch.float64, F16_O16: torch.float16, BF16: torch.bfloat16}.get(_fmt(fmt), torch.float32)
    _need(out, "out", gather_dtype, int(idx.numel()), stream=stream)
    d = len(cores)
    ptrs = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores])
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    _check(load().tt_gather(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dd, ctypes.c_void_p),
                            ctypes.cast(rr, ctypes.c_void_p), d, _fmt(fmt), _ptr(idx), int(idx.numel()),
                            _ptr(out), _stream(stream)))


def lrc_fro_diff(A, fa, B, fb, count: int, stream=None, want_norm: bool = True) -> Tuple[float, float]:
    """Returns (||A - B||_F, ||A||_F); B may be None.  With want_norm=False
    ||A||_F is not computed (NaN is returned in its place)."""
    if count > 0:
        _need(A, "A", storage_dtype(fa), count, stream=stream)
        if B is not None:
            _need(B, "B", storage_dtype(fb), count, stream=stream)
    diff = ctypes.c_double(0.0)
    norm = ctypes.c_double(float("nan"))
    _check(load().lrc_fro_diff(_ptr(A), _fmt(fa), _ptr(B), _fmt(fb) if B is not None else 0, count,
                               ctypes.addressof(diff), ctypes.addressof(norm) if want_norm else None,
                               _stream(stream)))
    return diff.value, norm.value


def lrc_fro_diff_noalloc(A, fa, B, fb, count: int, stream=None) -> Tuple[float, float]:
    """lrc_fro_diff without any device allocation (scratch is a fixed array
    inside the library); at most 268435456 elements.  Returns (||A - B||_F, ||A||_F)."""
    if count > 0:
        _need(A, "A", storage_dtype(fa), count, stream=stream)
        if B is not None:
            _need(B, "B", storage_dtype(fb), count, stream=stream)
    diff = ctypes.c_double(0.0)
    norm = ctypes.c_double(0.0)
    _check(load().lrc_fro_diff_noalloc(_ptr(A), _fmt(fa), _ptr(B), _fmt(fb) if B is not None else 0, count,
                                       ctypes.addressof(diff), ctypes.addressof(norm), _stream(stream)))
    return diff.value, norm.value


def lrc_lowrank_eta(U, S, Vt, Uh, Sh, Vht, fmt, m: int, n: int, k: int, stream=None,
                    want_norm: bool = True) -> Tuple[float, float]:
    """Returns (eta, ||U diag(s) V^T||_F) for binary64 factors U, S, Vt and the
    stored factors Uh, Sh, Vht of format fmt (layouts of lrc_apply).  With
    want_norm=False the norm is not returned (NaN in its place)."""
    eta = ctypes.c_double(0.0)
    norm = ctypes.c_double(float("nan"))
    if m > 0 and n > 0 and k > 0:
        import torch
        ldk, ldn, st = lrc_packed_ld(k), lrc_packed_ld(n), storage_dtype(fmt)
        for t, what, dt in ((U, "U", torch.float64), (Uh, "Uh", st)):
            _need(t, what, dt, _extent(m, k, ldk), stream=stream)
        for t, what, dt in ((S, "S", torch.float64), (Sh, "Sh", st)):
            _need(t, what, dt, k, stream=stream)
        for t, what, dt in ((Vt, "Vt", torch.float64), (Vht, "Vht", st)):
            _need(t, what, dt, _extent(k, n, ldn), stream=stream)
    _check(load().lrc_lowrank_eta(_ptr(U), _ptr(S), _ptr(Vt), _ptr(Uh), _ptr(Sh), _ptr(Vht), _fmt(fmt),
                                  m, n, k, ctypes.addressof(eta),
                                  ctypes.addressof(norm) if want_norm else None, _stream(stream)))
    return eta.value, norm.value


def lrc_tt_eta(cores: Sequence, cores_hat: Sequence, dims: Sequence[int], ranks: Sequence[int], fmt,
               stream=None, want_norm: bool = True) -> Tuple[float, float]:
    """Returns (eta_TT, ||T||_F) for binary64 cores and stored cores of format fmt."""
    import torch
    d = len(cores)
    shaped = len(dims) == d and len(ranks) == d + 1 and all(int(x) > 0 for x in list(dims) + list(ranks))
    for l, c in enumerate(cores):
        _need(c, f"cores[{l}]", torch.float64,
              int(ranks[l]) * int(dims[l]) * int(ranks[l + 1]) if shaped else 0, stream=stream)
    if len(cores_hat) == d:
        _need_cores(cores_hat, dims, ranks, fmt, stream)
    d = len(cores)
    if len(cores_hat) != d:
        raise ValueError("cores and cores_hat differ in length")
    p64 = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores])
    ph = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores_hat])
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    eta = ctypes.c_double(0.0)
    norm = ctypes.c_double(float("nan"))
    _check(load().lrc_tt_eta(ctypes.cast(p64, ctypes.c_void_p), ctypes.cast(ph, ctypes.c_void_p),
                             ctypes.cast(dd, ctypes.c_void_p), ctypes.cast(rr, ctypes.c_void_p), d, _fmt(fmt),
                             ctypes.addressof(eta), ctypes.addressof(norm) if want_norm else None,
                             _stream(stream)))
    return eta.value, norm.value


def lrc_certified(e_base: float, e_aug: float, eta: float) -> bool:
    return bool(load().lrc_certified(float(e_base), float(e_aug), float(eta)))


def lrc_tail_error(sigma, k: int) -> float:
    import numpy as np
    s = np.ascontiguousarray(sigma, dtype=np.float64)
    return float(load().lrc_tail_error(s.ctypes.data, s.size, int(k)))


def lrc_matrix_storage_ratio(m: int, n: int, k_base: int, k_aug: int, fmt) -> float:
    return float(load().lrc_matrix_storage_ratio(m, n, k_base, k_aug, _fmt(fmt)))


def lrc_tt_storage_bytes(dims: Sequence[int], ranks: Sequence[int], fmt) -> float:
    d = len(dims)
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    return float(load().lrc_tt_storage_bytes(ctypes.cast(dd, ctypes.c_void_p),
                                             ctypes.cast(rr, ctypes.c_void_p), d, _fmt(fmt)))


def lrc_launch_count() -> int:
    return int(load().lrc_launch_count())


def lrc_shutdown() -> None:
    _check(load().lrc_shutdown())


def lrc_device_status(stream=None) -> int:
    """Synchronises the stream; returns the lrc_status (0, or -6 if a bounded
    device wait gave up since the last call).  Does not raise."""
    return int(load().lrc_device_status(_stream(stream)))


def lrc_tt_svd(T, dims: Sequence[int], ranks: Sequence[int], cores: Sequence, stream=None,
               want_spectra: bool = False):
    """TT-SVD of the dense binary64 tensor T into `cores` (preallocated
    binary64 tensors of shapes ranks[l] x dims[l] x ranks[l+1]).  Returns
    (delta2, spectra): the discarded squared singular values per bond and,
    if asked, every bond's singular values (a list of arrays)."""
    import numpy as np
    import torch
    d = len(dims)
    if len(cores) != d or len(ranks) != d + 1:
        raise ValueError("cores needs d entries and ranks d + 1")
    _need(T, "T", torch.float64, np_prod(dims), stream=stream)
    _need_cores(cores, dims, ranks, "f64", stream)
    sizes, rest = [], np_prod(dims)
    for l in range(d - 1):
        rest //= int(dims[l])
        sizes.append(min(int(ranks[l]) * int(dims[l]), rest))
    delta2 = (ctypes.c_double * max(d - 1, 1))()
    spec = (ctypes.c_double * max(sum(sizes), 1))() if want_spectra else None
    ptrs = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores])
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    _check(load().lrc_tt_svd(_ptr(T), ctypes.cast(dd, ctypes.c_void_p), ctypes.cast(rr, ctypes.c_void_p), d,
                             ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(delta2, ctypes.c_void_p),
                             ctypes.cast(spec, ctypes.c_void_p) if spec is not None else None, _stream(stream)))
    spectra = None
    if spec is not None:
        flat, spectra, o = np.array(spec[:]), [], 0
        for n in sizes:
            spectra.append(flat[o:o + n])
            o += n
    return [delta2[i] for i in range(d - 1)], spectra


def lrc_tt_left_orthogonalize(cores: Sequence, dims: Sequence[int], ranks: Sequence[int], stream=None) -> None:
    """Left-orthogonal gauge of binary64 cores, in place."""
    d = len(cores)
    _need_cores(cores, dims, ranks, "f64", stream)
    ptrs = (ctypes.c_void_p * d)(*[c.data_ptr() for c in cores])
    dd = (ctypes.c_int64 * d)(*[int(x) for x in dims])
    rr = (ctypes.c_int64 * (d + 1))(*[int(x) for x in ranks])
    _check(load().lrc_tt_left_orthogonalize(ctypes.cast(ptrs, ctypes.c_void_p), ctypes.cast(dd, ctypes.c_void_p),
                                            ctypes.cast(rr, ctypes.c_void_p), d, _stream(stream)))


PROBE_KINDS = {"ffma": 0, "ffma2": 1, "dfma": 2, "dmma": 3}


def lrc_probe_peak(kind, iters: int, stream=None) -> float:
    """Measured flop/s of one arithmetic unit (kind: ffma, ffma2, dfma, dmma)."""
    k = PROBE_KINDS[kind] if isinstance(kind, str) else int(kind)
    out = ctypes.c_double(0.0)
    _check(load().lrc_probe_peak(k, int(iters), ctypes.addressof(out), _stream(stream)))
    return out.value


def lrc_selftest_wait_timeout(limit_ns: int, stream=None) -> None:
    _check(load().lrc_selftest_wait_timeout(int(limit_ns), _stream(stream)))


# --------------------------------------------------------------------------
# convenience helpers built only from the entry points above
# --------------------------------------------------------------------------

def round_matrix(src64, fmt, ld: Optional[int] = None, stream=None):
    """Round a 2-D CUDA float64 tensor into a new packed tensor (lrc_round_factors)."""
    import torch
    rows, cols = src64.shape
    if src64.stride(1) != 1 or (rows > 1 and src64.stride(0) < cols):
        src64 = src64.contiguous()
    ld_src = src64.stride(0) if rows > 1 else cols   # a single row may carry any stride
    ld = lrc_packed_ld(cols) if ld is None else ld
    dst = torch.empty((rows, ld), dtype=storage_dtype(fmt), device=src64.device)
    lrc_round_factors(src64, rows, cols, ld_src, dst, ld, fmt, stream)
    return dst


def widen_matrix(src, fmt, cols: int, stream=None):
    """Exact float64 copy (rows x packed ld) of a packed tensor (lrc_widen_factors)."""
    import torch
    rows, ld = src.shape
    dst = torch.empty((rows, lrc_packed_ld(cols)), dtype=torch.float64, device=src.device)
    lrc_widen_factors(src, fmt, rows, cols, ld, dst, dst.shape[1], stream)
    return dst
