"""GPU parity of the verification step (C ABI, sm_103a) against the CPU oracle.

Every test here calls libspecdiff through the C ABI on cuda:0 and compares with
oracle/ on the same seeded inputs (tolerances in tests/gpu_helpers.py).
"""
import math

import numpy as np
import pytest
import torch
from scipy import stats

import workloads as W
from oracle import philox as OP
from oracle import verify as OV
from gpu_helpers import compare, oracle_for, philox_words, run_gpu

pytestmark = pytest.mark.gpu

MODES = [("sample", OV.MODE_SAMPLE), ("block", OV.MODE_BLOCK)]


@pytest.fixture(scope="module")
def api():
    import __graft_entry__ as g
    g.build()
    from paper_2606_13426_gb300 import api as A
    return A


# ------------------------------------------------------------------ a1: RNG
def test_philox_bit_exact(api):
    rng = np.random.Generator(np.random.PCG64(1))
    ctr = rng.integers(0, 2 ** 32, size=(4096, 4), dtype=np.uint64).astype(np.uint32)
    ctr[:3] = [[0, 0, 0, 0], [0xFFFFFFFF] * 4, [0x243f6a88, 0x85a308d3, 0x13198a2e, 0x03707344]]
    for seed in (0, 0xFFFFFFFFFFFFFFFF, 0x299f31d0a4093822, 12345):
        got = api.philox(torch.from_numpy(ctr.view(np.int32)).cuda(), seed).cpu().numpy()
        np.testing.assert_array_equal(got.view(np.uint32), philox_words(ctr.astype(np.uint64), seed))


@pytest.mark.parametrize("stream", [OP.STREAM_RESID, OP.STREAM_BONUS, OP.STREAM_DRAFT])
def test_normals_match_oracle(api, stream):
    for Bn, d, seed in ((3, 4099, 7), (64, 1024, 2 ** 40 + 3)):
        got = api.normals(seed, Bn, d, stream, sub=2).cpu().numpy()
        ref = OP.normals(seed, np.arange(Bn), d, stream, sub=2)
        assert np.max(np.abs(got - ref)) < 4e-6


# ------------------------------------------------------------------ a4: U-sampler
def test_usample_matches_oracle(api):
    rng = np.random.Generator(np.random.PCG64(2))
    D, la, wb = [], [], []
    for Dv in (1e-3, 0.01, 0.1, 0.5, 1.0, 2.0, 4.0, 8.0, 16.0):
        for lav in (0.0, -1e-3, -0.1, -1.0, -5.0, -20.0):
            for w in [0, 1, 12345, 2 ** 31 - 1, 2 ** 31, 2 ** 32 - 2, 2 ** 32 - 1] + \
                    list(rng.integers(0, 2 ** 32, 9)):
                D.append(Dv); la.append(lav); wb.append(int(w))
    n_rand = 4000
    D += list(rng.uniform(0.02, 6.0, n_rand))
    la += list(-rng.exponential(1.0, n_rand) * (rng.uniform(size=n_rand) < 0.8))
    wb += list(rng.integers(0, 2 ** 32, n_rand))
    D = np.array(D, np.float32)
    la = np.array(la, np.float32)
    wb = np.array(wb, np.uint64).astype(np.uint32)
    U, st = api.usample(torch.from_numpy(D).cuda(), torch.from_numpy(la).cuda(),
                        torch.from_numpy(wb.view(np.int32)).cuda())
    U = U.cpu().numpy().astype(np.float64)
    assert np.all(st.cpu().numpy() == 0)
    Uo = OV.usample_bisection(D.astype(np.float64), la.astype(np.float64), OP.uniform_of(wb))
    err = np.abs(U - Uo)
    tol = 5e-6 + 3e-7 * np.abs(Uo)
    i = int(np.argmax(err - tol))
    assert np.all(err <= tol), "worst U error %g at D=%r la=%r w_bits=%d: gpu %r oracle %r" % (
        err[i], float(D[i]), float(la[i]), int(wb[i]), float(U[i]), float(Uo[i]))


def test_usample_degenerate_inputs(api):
    D = torch.tensor([0.0, -1.0, float("nan"), 1.0], device="cuda")
    la = torch.tensor([-1.0, -1.0, -1.0, float("nan")], device="cuda")
    w = torch.zeros(4, dtype=torch.int32, device="cuda")
    U, st = api.usample(D, la, w)
    st = st.cpu().numpy()
    assert st[0] == 1 and st[1] == 1 and st[2] == 2 and st[3] == 2
    assert torch.isnan(U).all()


def test_usample_range_of_the_bracket(api):
    """The bracket's candidates t = a+ - U reach s0 2^(255/8 - 8) with s0 = 1/max(1, |a-|)
    (the warp version s0 2^23), which covers the residual whenever |Delta| is below about
    5800 (at |Delta| = D and alpha = 1 the residual is close to N(0, 1) while a+ = D/2).
    Inside that range U matches the oracle (up to the rounding of a+ itself, from which U
    is formed in fp32); far outside it the kernel reports SDV_STATUS_USAMPLE_RANGE."""
    wbits = [1, 12345, 2 ** 31 - 1, 2 ** 31, 3 * 2 ** 30, 2 ** 32 - 2]
    D_in = [64.0, 512.0, 3000.0]
    la_in = [0.0, -5.0]
    D, la, wb = [], [], []
    for Dv in D_in:
        for lav in la_in:
            for w in wbits:
                D.append(Dv); la.append(lav); wb.append(w)
    n_in = len(D)
    for Dv in (2.0e4, 1.0e5):
        for w in wbits:
            D.append(Dv); la.append(0.0); wb.append(w)
    D = np.array(D, np.float32)
    la = np.array(la, np.float32)
    wb = np.array(wb, np.uint64).astype(np.uint32)
    U, st = api.usample(torch.from_numpy(D).cuda(), torch.from_numpy(la).cuda(),
                        torch.from_numpy(wb.view(np.int32)).cuda())
    U = U.cpu().numpy().astype(np.float64)
    st = st.cpu().numpy()
    assert np.all(st[:n_in] == 0)
    Uo = OV.usample_bisection(D[:n_in].astype(np.float64), la[:n_in].astype(np.float64),
                              OP.uniform_of(wb[:n_in]))
    ap = la[:n_in] / D[:n_in] + 0.5 * D[:n_in]
    tol = 5e-6 + 3e-7 * np.abs(Uo) + 2.0 ** -23 * np.abs(ap)
    assert np.all(np.abs(U[:n_in] - Uo) <= tol), np.max(np.abs(U[:n_in] - Uo) / tol)
    assert np.all(st[n_in:] & 4), st[n_in:]          # SDV_STATUS_USAMPLE_RANGE
    assert np.all(np.isfinite(U[n_in:]))


# ------------------------------------------------------------------ a2: log ratios
@pytest.mark.parametrize("kind,B,L,d", [("tiny", 4, 4, 16), ("pixel", 32, 8, 3072),
                                        ("latent", 8, 16, 16384), ("pixel", 5, 3, 4099),
                                        ("pixel", 7, 5, 1), ("latent", 3, 2, 1001),
                                        ("highres", 2, 4, 196608)])
def test_log_ratios_match_oracle(api, kind, B, L, d):
    inp = W.make_verify_inputs(kind, B=B, L=L, d=d, per_chain_sigma=True)
    from gpu_helpers import to_dev
    Leff = np.random.Generator(np.random.PCG64(B)).integers(0, L + 1, B).astype(np.int32)
    lr, dn = api.log_ratios(to_dev(inp, "x_draft"), to_dev(inp, "mu_target"),
                            to_dev(inp, "mu_draft"), torch.from_numpy(inp["sigma"]).cuda(),
                            L_eff=torch.from_numpy(Leff).cuda())
    ell_o, dn_o = OV.log_ratios(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"])
    mask = np.arange(L)[None, :] < Leff[:, None]
    ell_o = np.where(mask, ell_o, 0.0)
    dn_o = np.where(mask, dn_o, 0.0)
    lr, dn = lr.cpu().numpy(), dn.cpu().numpy()
    assert np.all(np.abs(lr - ell_o) <= 1e-5 * np.maximum(1.0, np.abs(ell_o)))
    assert np.all(np.abs(dn - dn_o) <= 1e-5 * np.maximum(1.0, dn_o))


# ------------------------------------------------------------------ a3: acceptance scan
@pytest.mark.parametrize("mode,m", MODES)
@pytest.mark.parametrize("L", [1, 4, 31, 32, 33, 64])
def test_accept_scan_matches_oracle(api, mode, m, L):
    rng = np.random.Generator(np.random.PCG64(L))
    n = 3000
    ell = rng.normal(-0.4, 1.2, (n, L)).astype(np.float32)
    ell[rng.uniform(size=(n, L)) < 0.1] = 0.0
    dn = rng.uniform(0.0, 3.0, (n, L)).astype(np.float32)
    dn[rng.uniform(size=(n, L)) < 0.02] = 0.0
    Leff = rng.integers(0, L + 1, n).astype(np.int32)
    for omega in (1.0, 1.7):
        tau, la = api.accept_scan(torch.from_numpy(ell).cuda(), torch.from_numpy(dn).cuda(), 99,
                                  mode, torch.from_numpy(Leff).cuda(), omega)
        tau, la = tau.cpu().numpy(), la.cpu().numpy()
        eta = OP.coins(99, np.arange(n), L)
        if m == OV.MODE_SAMPLE:
            to = OV.sample_verification(ell, eta, Leff, omega)
            lao = np.zeros(n)
            h = None
        else:
            to, lao, _, h = OV.block_verification(ell, dn, eta, Leff, omega)
        to = np.where(Leff == 0, 0, to)
        o = dict(ell=ell.astype(np.float64) * np.where(np.arange(L) < Leff[:, None], 1, 0),
                 eta=eta, h=h, dnorm=dn.astype(np.float64))
        from gpu_helpers import near_tie
        diff = tau != to
        assert np.all(near_tie(o, m, omega, rtol=1e-6)[diff]), np.nonzero(diff)[0][:5]
        assert diff.mean() < 0.01
        same = ~diff & (Leff > 0)
        assert np.all(np.abs(la[same] - lao[same]) <= 1e-5 * np.maximum(1, np.abs(lao[same])) + 1e-6)


# ------------------------------------------------------------------ a1-a5: whole step
@pytest.mark.parametrize("mode,m", MODES)
@pytest.mark.parametrize("kind,B,L,d", [("tiny", 4, 4, 16), ("tiny", 64, 4, 16),
                                        ("pixel", 64, 8, 3072), ("latent", 16, 16, 16384),
                                        ("pixel", 48, 6, 4101), ("latent", 24, 5, 1003),
                                        ("highres", 2, 32, 196608)])
def test_verify_matches_oracle(api, mode, m, kind, B, L, d):
    inp = W.make_verify_inputs(kind, B=B, L=L, d=d)
    g = run_gpu(api, inp, 1234, mode)
    o = oracle_for(inp, 1234, m)
    compare(g, o, m, inp["dtype"])
    # the residual's 1-D draw agrees where both sides drew one
    both = np.isfinite(g["aux"][:, 0]) & np.isfinite(o["U"]) & (g["accepted_len"] == o["accepted_len"])
    assert np.all(np.abs(g["aux"][both, 0] - o["U"][both]) <= 5e-6 + 3e-7 * np.abs(o["U"][both]))


@pytest.mark.parametrize("kind,sample", [("pixel", None), ("latent", 16), ("highres", 3)])
@pytest.mark.parametrize("mode,m", MODES)
def test_verify_full_size_sampled(api, kind, sample, mode, m):
    """The full workload sizes on the GPU, the oracle on a sample of chains (chains are independent)."""
    inp = W.make_verify_inputs(kind)
    g = run_gpu(api, inp, 2024, mode)
    Bn = inp["B"]
    chains = np.arange(Bn) if sample is None else \
        np.random.Generator(np.random.PCG64(5)).choice(Bn, sample, replace=False)
    o = oracle_for(inp, 2024, m, chains=chains)
    gs = {k: v[chains] for k, v in g.items()}
    compare(gs, o, m, inp["dtype"], max_tie_frac=0.1)


# Many chains (B >= 512) take the two-kernel path: k_tiles streams, k_finish finishes
# every chain with one warp (its own U-sampler and residual writer).
@pytest.mark.parametrize("mode,m", MODES)
@pytest.mark.parametrize("kind,B,L,d,sample", [("tiny", 600, 8, 64, None), ("latent", 520, 4, 1003, None),
                                               ("pixel", 512, 3, 5000, 64), ("pixel", 1024, 16, 1024, 96)])
def test_verify_many_chains_matches_oracle(api, mode, m, kind, B, L, d, sample):
    inp = W.make_verify_inputs(kind, B=B, L=L, d=d)
    g = run_gpu(api, inp, 4321, mode)
    chains = np.arange(B) if sample is None else \
        np.random.Generator(np.random.PCG64(6)).choice(B, sample, replace=False)
    o = oracle_for(inp, 4321, m, chains=chains)
    gs = {k: v[chains] for k, v in g.items()}
    compare(gs, o, m, inp["dtype"])
    both = np.isfinite(gs["aux"][:, 0]) & np.isfinite(o["U"]) & (gs["accepted_len"] == o["accepted_len"])
    assert both.sum() > 0
    assert np.all(np.abs(gs["aux"][both, 0] - o["U"][both]) <= 5e-6 + 3e-7 * np.abs(o["U"][both]))


def test_verify_many_chains_ragged_bonus_reflection(api):
    Bn = 640
    inp = W.make_verify_inputs("pixel", B=Bn, L=6, d=300, per_chain_sigma=True)
    rng = np.random.Generator(np.random.PCG64(18))
    Leff = rng.integers(0, 7, Bn).astype(np.int32)
    Leff[:3] = [0, 1, 6]
    mqb = rng.standard_normal((Bn, 300)).astype(np.float32)
    sb = rng.uniform(0.1, 1.0, Bn).astype(np.float32)
    for mode, m in MODES:
        g = run_gpu(api, inp, 78, mode, L_eff=Leff, mu_target_bonus=mqb, sigma_bonus=sb)
        o = oracle_for(inp, 78, m, Leff=Leff, mu_target_bonus=mqb, sigma_bonus=sb)
        assert np.all(g["accepted_len"][Leff == 0] == 0)
        compare(g, o, m, "f32")
    g = run_gpu(api, inp, 79, "sample", residual="reflection")
    o = oracle_for(inp, 79, OV.MODE_SAMPLE, residual=OV.RESIDUAL_REFLECTION)
    compare(g, o, OV.MODE_SAMPLE, "f32")


def test_verify_ragged_windows_bonus_and_inactive(api):
    inp = W.make_verify_inputs("pixel", B=40, L=6, d=1000, per_chain_sigma=True)
    rng = np.random.Generator(np.random.PCG64(8))
    Leff = rng.integers(0, 7, 40).astype(np.int32)
    Leff[:3] = [0, 1, 6]
    mqb = rng.standard_normal((40, 1000)).astype(np.float32)
    sb = rng.uniform(0.1, 1.0, 40).astype(np.float32)
    for mode, m in MODES:
        g = run_gpu(api, inp, 77, mode, L_eff=Leff, mu_target_bonus=mqb, sigma_bonus=sb)
        o = oracle_for(inp, 77, m, Leff=Leff, mu_target_bonus=mqb, sigma_bonus=sb)
        assert np.all(g["accepted_len"][Leff == 0] == 0)
        compare(g, o, m, "f32")


def test_verify_reflection_residual(api):
    inp = W.make_verify_inputs("pixel", B=64, L=8, d=3072)
    g = run_gpu(api, inp, 5, "sample", residual="reflection")
    o = oracle_for(inp, 5, OV.MODE_SAMPLE, residual=OV.RESIDUAL_REFLECTION)
    compare(g, o, OV.MODE_SAMPLE, "f32")


@pytest.mark.parametrize("omega", [0.5, 2.0])
@pytest.mark.parametrize("mode,m", MODES)
def test_verify_temperature(api, omega, mode, m):
    inp = W.make_verify_inputs("pixel", B=64, L=8, d=2048)
    g = run_gpu(api, inp, 9, mode, omega=omega)
    o = oracle_for(inp, 9, m, omega=omega)
    compare(g, o, m, "f32", omega=omega)


def test_verify_edge_shapes(api):
    # B = 1, L = 1, d = 1 and odd sizes; equal means accept everything
    for (Bn, L, d) in ((1, 1, 1), (1, 1, 5), (3, 64, 7), (2, 33, 17)):
        inp = W.make_verify_inputs("tiny", B=Bn, L=L, d=d)
        for mode, m in MODES:
            compare(run_gpu(api, inp, 3, mode), oracle_for(inp, 3, m), m, "f32")
    inp = W.make_verify_inputs("tiny", B=6, L=5, d=9)
    inp["mu_target"] = inp["mu_draft"].copy()
    for mode, m in MODES:
        g = run_gpu(api, inp, 3, mode)
        assert np.all(g["accepted_len"] == 5)
        np.testing.assert_array_equal(g["y"], inp["x_draft"][:, -1])


def test_zero_delta_step_is_never_the_residual(api):
    """A step with m^p = m^q is never rejected: in sample mode its ratio is 1, and in block
    mode h_{j-1} = 0 unless alpha_{j-1} = 1, in which case alpha_j = 1 and h_j = 1.  So the
    SDV_STATUS_ZERO_DELTA branch (y = m^q + sigma G) is unreachable for exact zeros."""
    rng = np.random.Generator(np.random.PCG64(10))
    Bn, L, d = 4000, 3, 4
    s = np.full((Bn, L), 0.5, np.float32)
    mp = rng.standard_normal((L, d)).astype(np.float32)
    mq = mp.copy()
    e = rng.standard_normal((L, d))
    e /= np.linalg.norm(e, axis=1, keepdims=True)
    mq[0] -= (0.5 * 2.5 * e[0]).astype(np.float32)
    mq[2] -= (0.5 * 2.5 * e[2]).astype(np.float32)
    x = (mp[None] + 0.5 * rng.standard_normal((Bn, L, d))).astype(np.float32)
    inp = dict(x_draft=x, mu_target=np.broadcast_to(mq, x.shape).copy(),
               mu_draft=np.broadcast_to(mp, x.shape).copy(), sigma=s, dtype="f32")
    for mode, m in MODES:
        g = run_gpu(api, inp, 4, mode)
        o = oracle_for(inp, 4, m)
        compare(g, o, m, "f32")
        assert not np.any(g["accepted_len"] == 1)      # tau = 2 would be the zero-delta step
        assert not np.any(g["status"] & 1)


# ------------------------------------------------------------------ statistics on the GPU path
@pytest.mark.parametrize("mode", ["sample", "block"])
def test_gpu_single_step_output_follows_target(api, mode):
    rng = np.random.Generator(np.random.PCG64(12))
    Bn, d, sigma, D = 200_000, 3, 0.6, 1.1
    e = rng.standard_normal(d)
    e /= np.linalg.norm(e)
    mp = rng.standard_normal(d).astype(np.float32)
    mq = (mp - sigma * D * e).astype(np.float32)
    x = (mp + sigma * rng.standard_normal((Bn, 1, d))).astype(np.float32)
    inp = dict(x_draft=x, mu_target=np.broadcast_to(mq, x.shape).copy(),
               mu_draft=np.broadcast_to(mp, x.shape).copy(),
               sigma=np.full((Bn, 1), sigma, np.float32), dtype="f32")
    g = run_gpu(api, inp, 31, mode)
    z = (g["y"] - mq) / sigma
    assert stats.kstest(z @ e, "norm").pvalue > 1e-3
    acc = np.mean(g["accepted_len"] == 1)
    p = 2 * stats.norm.cdf(-D / 2)
    assert abs(acc - p) < 4 * math.sqrt(p * (1 - p) / Bn)


def test_gpu_block_beats_sample_in_expectation(api):
    inp = W.make_verify_inputs("pixel")
    taus = {}
    for mode in ("sample", "block"):
        t = [run_gpu(api, inp, s, mode)["accepted_len"] + 1 for s in range(8)]
        taus[mode] = np.concatenate(t).astype(np.float64)
    assert taus["block"].mean() > taus["sample"].mean()


# ------------------------------------------------------------------ special functions
def test_device_special_functions(api):
    """The kernels' own erfcx (a polynomial fit, gen_erfcx_coeffs.py), log Phi and
    g' = lambda + z against scipy in fp64 over the ranges the acceptance rule and the
    U-sampler reach, including the negative side of erfcx and both forms of g'."""
    from scipy.special import erfcx, log_ndtr
    z = np.concatenate([np.linspace(-9.0, 30.0, 20001), [0.0, 1e-8, 1e3, 1e6]]).astype(np.float32)
    zz = torch.from_numpy(z).cuda()
    z64 = z.astype(np.float64)
    e = api.special("erfcx", zz).cpu().numpy().astype(np.float64)
    ref = erfcx(z64)
    fin = np.isfinite(ref)
    assert np.max(np.abs(e[fin] / ref[fin] - 1.0)) < 6e-7
    ln = api.special("log_ndtr", torch.from_numpy(np.linspace(-30, 8, 20001).astype(np.float32)).cuda())
    x = np.linspace(-30, 8, 20001).astype(np.float32).astype(np.float64)
    lr = log_ndtr(x)
    err = np.abs(ln.cpu().numpy() - lr)
    assert np.all(err <= 4e-7 * np.maximum(1.0, np.abs(lr)))
    s = np.linspace(-60.0, 12.0, 20001).astype(np.float32)
    gp = api.special("gprime", torch.from_numpy(s).cuda()).cpu().numpy().astype(np.float64)
    s64 = s.astype(np.float64)
    lam = np.exp(-0.5 * s64 * s64 - 0.5 * np.log(2 * np.pi) - log_ndtr(s64))
    gref = lam + s64
    assert np.all(np.abs(gp - gref) <= 1e-6 * np.maximum(1.0, np.abs(gref)) + 4e-7 * np.abs(s64))
