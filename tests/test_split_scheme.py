"""The arithmetic scheme of the FP32 tensor-core variant (LRC_F32_TC),
emulated in numpy on the CPU: binary32 values scaled by a power of two per
group (largest magnitude into [2^14, 2^15)) and split into binary16 parts
hi = fp16(x), lo = fp16(x - hi) keep about 22 bits of the group's scale,
and the three products W_hi U_hi + W_lo U_hi + W_hi U_lo stay within the
binary32 tolerance of the exact product."""
import numpy as np


def group_exp(maxabs):
    if not (maxabs > 0) or not np.isfinite(maxabs):
        return 0
    e = 14 - int(np.floor(np.log2(np.float32(maxabs))))
    return int(np.clip(e, -60, 60))


def split(x32, group_rows):
    """Parts of a binary32 matrix, scaled per group of rows (1 = per row)."""
    hi = np.empty(x32.shape, np.float16)
    lo = np.empty(x32.shape, np.float16)
    ex = np.empty(x32.shape[0], np.int64)
    for r0 in range(0, x32.shape[0], group_rows):
        g = x32[r0:r0 + group_rows]
        e = group_exp(float(np.max(np.abs(g))))
        y = (g * np.float32(2.0 ** e)).astype(np.float32)          # exact: a power of two
        h = y.astype(np.float16)
        l = (y - h.astype(np.float32)).astype(np.float16)          # residual exact in binary32
        hi[r0:r0 + group_rows], lo[r0:r0 + group_rows], ex[r0:r0 + group_rows] = h, l, e
    return hi, lo, ex


def test_parts_keep_22_bits_of_the_group_scale():
    rng = np.random.default_rng(5)
    x = (rng.standard_normal((256, 96)) * np.exp2(rng.integers(-40, 40, size=(256, 1)))).astype(np.float32)
    for group in (1, 32):
        hi, lo, ex = split(x, group)
        back = (hi.astype(np.float64) + lo.astype(np.float64)) * np.exp2(-ex.astype(np.float64))[:, None]
        for r0 in range(0, 256, group):
            g = slice(r0, r0 + group)
            scale = np.max(np.abs(x[g].astype(np.float64)))
            assert np.max(np.abs(back[g] - x[g])) <= 2.0 ** -22 * scale


def test_scaling_is_what_keeps_the_bits():
    """A group of magnitude about 1e-3 split without the power-of-two scale
    leaves lo among the binary16 subnormals (absolute step 2^-24) and keeps
    only about 17 bits of the group's scale; scaled, it keeps 22."""
    rng = np.random.default_rng(7)
    x = (rng.standard_normal((32, 64)) * 1e-3).astype(np.float32)
    scale = np.max(np.abs(x.astype(np.float64)))
    h = x.astype(np.float16)
    l = (x - h.astype(np.float32)).astype(np.float16)
    err_plain = np.max(np.abs(h.astype(np.float64) + l.astype(np.float64) - x))
    hi, lo, ex = split(x, 32)
    back = (hi.astype(np.float64) + lo.astype(np.float64)) * np.exp2(-float(ex[0]))
    err_scaled = np.max(np.abs(back - x))
    assert err_plain > 2.0 ** -18 * scale
    assert err_scaled <= 2.0 ** -22 * scale
    assert err_plain >= 16 * err_scaled


def test_three_products_meet_the_binary32_tolerance():
    rng = np.random.default_rng(6)
    b, m, k = 64, 200, 136
    W = (rng.standard_normal((b, k)) * np.exp2(rng.integers(-20, 20, size=(b, 1)))).astype(np.float32)
    U = rng.standard_normal((m, k)).astype(np.float32)
    Wh, Wl, ew = split(W, 1)
    Uh, Ul, eu = split(U, 32)
    f = lambda a: a.astype(np.float64)                                 # noqa: E731
    Y = (f(Wh) @ f(Uh).T + f(Wl) @ f(Uh).T + f(Wh) @ f(Ul).T)
    Y *= np.exp2(-ew.astype(np.float64))[:, None] * np.exp2(-eu.astype(np.float64))[None, :]
    exact = f(W) @ f(U).T
    rel = np.linalg.norm(Y - exact, axis=1) / np.linalg.norm(exact, axis=1)
    assert rel.max() <= 1e-6, rel.max()
    # the dropped term W_lo U_lo is below 2^-22 of the product's scale
    assert np.max(np.abs(f(Wl) @ f(Ul).T)) <= 2.0 ** -22 * np.max(np.abs(f(Wh) @ f(Uh).T)) * 4
