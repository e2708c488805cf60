"""bfloat16 storage (LRC_BF16; Sec. 3.2 precision table) through every entry
point: bit-exact rounding and exact widening, the apply and the TT
reconstruction against the oracle on the same rounded inputs, the Frobenius
difference, the fused eta and the sampled entries.

Tolerance of the apply and TT (parity.TOL["bf16"] = 4 u, u = 2^-8): products
of bfloat16 numbers are exact in binary32 and accumulate in binary32 (about
1e-6 relative at these sizes); the intermediate W (or the TT chain's Z) and
the output are each rounded once to bfloat16, which moves an orthonormal
product by at most about u each: 2u in all, with a factor-two margin."""
import numpy as np
import pytest
import torch

import oracle
import workloads as W
from parity import TOL, bits, oracle_inputs, packed, rel_fro, to_dev

pytestmark = pytest.mark.gpu

F = "bf16"


def bf16_values(b):
    return (np.asarray(b, dtype=np.uint32) << 16).view(np.float32).astype(np.float64)


def gpu_round_flat(lrc, x, dev):
    out = lrc.round_matrix(to_dev(x.reshape(1, -1), dev), F, ld=x.size)
    torch.cuda.synchronize()
    return bits(out, F).reshape(-1)


def test_round_midpoints_and_thresholds_bit_exact(lrc, cuda):
    pos = np.arange(0, 0x7F80, dtype=np.uint16)
    lo, hi = bf16_values(pos[:-1]), bf16_values(pos[1:])
    mid = (lo + hi) / 2.0
    bmax = (2.0 - 2.0 ** -7) * 2.0 ** 127
    x = np.concatenate([lo, mid, np.nextafter(mid, np.inf), np.nextafter(mid, -np.inf), -mid,
                        [bmax, (2.0 - 2.0 ** -8) * 2.0 ** 127, 1e300, -1e300, 5e-324, 2.0 ** -134, -0.0, 0.0,
                         np.inf, -np.inf, 1.0 + 2.0 ** -8 + 2.0 ** -40]])
    assert np.array_equal(gpu_round_flat(lrc, x, cuda), oracle.round_bits(x, F))


def test_round_wide_range_and_nan(lrc, cuda):
    rng = np.random.default_rng(21)
    x = rng.standard_normal(1_000_003) * np.exp2(rng.uniform(-150, 130, 1_000_003))
    assert np.array_equal(gpu_round_flat(lrc, x, cuda), oracle.round_bits(x, F))
    dec = oracle.decode(gpu_round_flat(lrc, np.array([np.nan, -np.nan, 2.0]), cuda), F)
    assert np.isnan(dec[:2]).all() and dec[2] == 2.0


@pytest.mark.parametrize("rows,cols,ld_src", [(1, 1, 1), (7, 33, 33), (5, 34, 40), (64, 512, 512)])
def test_packing_padding_and_exact_widening(lrc, cuda, rows, cols, ld_src):
    src = W.gaussian((rows, ld_src), rows * 7 + cols)
    ld = lrc.lrc_packed_ld(cols)
    dst = torch.full((rows, ld), 7, dtype=torch.bfloat16, device=cuda)
    lrc.lrc_round_factors(to_dev(src, cuda), rows, cols, ld_src, dst, ld, F)
    want = oracle.round_pack(src[:, :cols], F, ld=ld)
    assert np.array_equal(bits(dst, F), want)
    wide = lrc.widen_matrix(dst, F, cols)
    assert np.array_equal(wide.cpu().numpy()[:, :cols], oracle.decode(want[:, :cols], F))


def run_apply(lrc, dev, U, s, Vt, X):
    m, k = U.shape
    n = Vt.shape[1]
    b = X.shape[0]
    Ud, Sd, Vd, Xd = (packed(lrc, a, F, dev) for a in (U, s, Vt, X))
    Y = torch.full((b, m), float("nan"), dtype=torch.bfloat16, device=dev)
    lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, F)
    assert lrc.lrc_device_status() == 0
    return Y.double().cpu().numpy()


@pytest.mark.parametrize("m,n,k,b", [
    (512, 512, 34, 64), (100, 300, 1, 1), (257, 129, 19, 1), (333, 1031, 37, 5), (48, 40, 60, 5),
    (777, 1029, 272, 250), (2048, 1536, 144, 300), (1000, 5000, 272, 16),
])
def test_apply_vs_oracle(lrc, cuda, m, n, k, b):
    f = W.random_factors(m, n, k, seed=m + 2 * n + k)
    X = W.gaussian((b, n), b + 9)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X)
    want = oracle.apply(*oracle_inputs(f.U, f.s, f.Vt, X, F))
    assert rel_fro(got, want) <= TOL[F]


def test_apply_integer_inputs_exact(lrc, cuda):
    # small integers: products and sums are exact in binary32, W = X V diag(s)
    # stays an integer below 2^8 (exact in bfloat16), and so does Y
    m, n, k, b = 130, 40, 6, 17
    U = W.integer_valued((m, k), 1, -1, 1)
    s = W.integer_valued((k,), 2, 1, 1)
    Vt = W.integer_valued((k, n), 3, -1, 1)
    X = W.integer_valued((b, n), 4, -1, 1)
    want = oracle.apply(U, s, Vt, X)
    assert np.max(np.abs(oracle.apply(np.eye(k), s, Vt, X))) < 256 and np.max(np.abs(want)) < 256
    assert np.array_equal(run_apply(lrc, cuda, U, s, Vt, X), want)


def test_apply_large_workload_sampled_rows(lrc, cuda):
    cfg = W.MATRIX_CONFIGS["large"]
    f = W.matrix_factors(cfg, "f16")          # the binary16 rank set, k' = 144
    X = W.queries(cfg)
    got = run_apply(lrc, cuda, f.U, f.s, f.Vt, X)
    rows = W.sample_indices(256, cfg.b, 99)
    want = oracle.apply_rows(*oracle_inputs(f.U, f.s, f.Vt, X, F), rows)
    assert rel_fro(got[rows], want) <= TOL[F]
    assert np.isfinite(got).all()


@pytest.mark.parametrize("b", [1, 3000])
def test_apply_bitwise_reproducible(lrc, cuda, b):
    m, n, k = 700, 2100, 72
    f = W.random_factors(m, n, k, seed=b + 41)
    X = W.gaussian((b, n), b + 42)
    Ud, Sd, Vd, Xd = (packed(lrc, a, F, cuda) for a in (f.U, f.s, f.Vt, X))
    outs = []
    for _ in range(2):
        Y = torch.empty((b, m), dtype=torch.bfloat16, device=cuda)
        lrc.lrc_apply(Ud, Sd, Vd, Xd, Y, m, n, k, b, F)
        torch.empty(1 << 22, device=cuda).uniform_()
        outs.append(Y.clone())
    assert torch.equal(outs[0].view(torch.int16), outs[1].view(torch.int16))


def run_tt(lrc, dev, cores64):
    rc = [oracle.rounded(c, F) for c in cores64]
    dc = [to_dev(c, dev).to(torch.bfloat16).contiguous() for c in rc]       # exact: values are bfloat16
    dims = [c.shape[1] for c in cores64]
    ranks = [1] + [c.shape[2] for c in cores64]
    out = torch.full((int(np.prod(dims)),), float("nan"), dtype=torch.bfloat16, device=dev)
    lrc.tt_reconstruct(dc, dims, ranks, F, out)
    assert lrc.lrc_device_status() == 0
    return out.double().cpu().numpy(), rc, dc


@pytest.mark.parametrize("dims,r,kind", [
    ((37, 29, 41), 9, "gauss_geo"),            # product chain with tensor-core output product
    ((8, 9, 7, 6, 5), 11, "gauss_alg"),
    ((16,) * 5, 28, "gauss_alg"),
    ((64, 48, 224), 70, "smooth"),             # rank above the chain's on-chip limit: CUDA-core chain
    ((300, 5), (1, 4, 1), None),
])
def test_tt_vs_oracle(lrc, cuda, dims, r, kind):
    if kind is None:
        cores = [W.gaussian((r[l], dims[l], r[l + 1]), 60 + l) for l in range(len(dims))]
    else:
        cores = W.make_tt(dims, W.capped_ranks(dims, r), kind, 17)
    got, rc, _ = run_tt(lrc, cuda, cores)
    want = oracle.tt_full(rc).reshape(-1)
    assert rel_fro(got, want) <= TOL[F]


@pytest.mark.parametrize("name", ["tt3", "tt6", "tt_hsi"])
def test_tt_workloads_sampled_entries(lrc, cuda, name):
    cfg = W.TT_CONFIGS[name]
    cores = W.tt_cores(cfg, "f16")            # the binary16 rank sets
    got, rc, dc = run_tt(lrc, cuda, cores)
    idx = W.sample_indices(20000, got.size, 3)
    assert rel_fro(got[idx], oracle.tt_entries(rc, idx)) <= TOL[F]
    assert np.isfinite(got).all()
    # sampled entries: one chain per entry, bfloat16 output
    ranks = [1] + [c.shape[2] for c in cores]
    didx = torch.from_numpy(idx.astype(np.int64)).to(cuda)
    g = torch.empty(idx.size, dtype=torch.bfloat16, device=cuda)
    lrc.tt_gather(dc, cfg.dims, ranks, F, didx, g)
    assert rel_fro(g.double().cpu().numpy(), oracle.tt_entries(rc, idx)) <= 2.0 ** -8


def test_fro_diff_with_bf16_operands(lrc, cuda):
    count = 333_335
    a = oracle.rounded(W.gaussian((count,), 1), F)
    b = oracle.rounded(W.gaussian((count,), 2), F)
    ta, tb = to_dev(a, cuda).to(torch.bfloat16), to_dev(b, cuda).to(torch.bfloat16)
    for A, fa, B, fb, x, y in ((ta, F, tb, F, a, b), (to_dev(a, cuda), "f64", tb, F, a, b)):
        d, na = lrc.lrc_fro_diff(A, fa, B, fb, count)
        wd, wna = oracle.fro_diff(x, y)
        assert abs(d - wd) <= 1e-12 * wd and abs(na - wna) <= 1e-12 * wna


def gamma(count: int) -> float:
    u = 2.0 ** -53
    return count * u / (1 - count * u)


@pytest.mark.parametrize("m,n,k", [(5, 4, 3), (300, 200, 33), (1000, 777, 144)])
def test_fused_eta_vs_oracle(lrc, cuda, m, n, k):
    f = W.random_factors(m, n, k, seed=m + n + k)
    f64 = [packed(lrc, a, "f64", cuda) for a in (f.U, f.s, f.Vt)]
    low = [packed(lrc, a, F, cuda) for a in (f.U, f.s, f.Vt)]
    eta, _ = lrc.lrc_lowrank_eta(*f64, *low, F, m, n, k)
    want = oracle.eta_matrix(f.U, f.s, f.Vt, F)
    bound = float(np.sum(np.abs(f.s) * np.linalg.norm(f.U, axis=0) * np.linalg.norm(f.Vt, axis=1)))
    assert abs(eta - want) <= 4 * gamma(k + 1) * bound + 1e-10 * want


def test_fused_eta_tt_vs_oracle(lrc, cuda):
    dims = (40, 36, 30)
    cores = W.make_tt(dims, W.capped_ranks(dims, 10), "gauss_geo", 8)
    ranks = [1] + [c.shape[2] for c in cores]
    c64 = [to_dev(c, cuda).contiguous() for c in cores]
    low = [lrc.round_matrix(c.reshape(1, -1), F, ld=c.numel()).reshape(c.shape) for c in c64]
    rc = [oracle.rounded(c, F) for c in cores]
    assert all(np.array_equal(lo.double().cpu().numpy(), r) for lo, r in zip(low, rc))
    eta, _ = lrc.lrc_tt_eta(c64, low, dims, ranks, F)
    want = oracle.eta_tt(cores, F)
    absT = oracle.tt_full([np.abs(c) for c in cores])
    assert abs(eta - want) <= 4 * gamma(sum(ranks) + len(dims)) * float(np.linalg.norm(absT)) + 1e-10 * want
