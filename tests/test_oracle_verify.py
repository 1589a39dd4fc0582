"""Pins for the fp64 verification oracle against what the paper and the mathematics fix.

Every check compares the oracle with something other than itself: closed forms
the paper proves (1 - TV acceptance, Lemma accept-prob, the residual mass v, the
alpha = 1 residual mean), library densities and quadrature, brute-force
enumeration of coin patterns, Gauss-Hermite integration over the draft noise,
and the exactness theorem (the emitted state follows the target kernel).
"""
import itertools
import math

import numpy as np
import pytest
from scipy import integrate, stats
from scipy.special import ndtr

from oracle import philox
from oracle import verify as V


def _unit(rng, d):
    e = rng.standard_normal(d)
    return e / np.linalg.norm(e)


def _perp(rng, e):
    z = rng.standard_normal(e.shape)
    z -= e * (z @ e)
    return z / np.linalg.norm(z)


def accept_prob_lemma(log_alpha, D, omega=1.0):
    """Lemma accept-prob: int p(y) min{1, alpha q^w(y)/p^w(y)} dy."""
    w2 = omega * omega
    A = w2 * log_alpha / D - D / 2.0
    return ndtr(A) + math.exp(log_alpha) * math.exp(D * D / (2 * w2) * (1.0 / w2 - 1.0)) * (
        1.0 - ndtr(A + D / w2))


# ---------------------------------------------------------------- log ratios
def test_log_ratio_closed_form_on_constructed_inputs():
    """x = m^p + sigma (u e + z_perp), m^q = m^p - sigma D e  =>  ell = -u D - D^2/2."""
    rng = np.random.Generator(np.random.PCG64(11))
    for d in (2, 16, 3072):
        for _ in range(5):
            sigma = rng.uniform(0.01, 2.0)
            D = rng.uniform(0.05, 5.0)
            u = rng.standard_normal()
            e = _unit(rng, d)
            zp = _perp(rng, e) * rng.uniform(0, 3 * math.sqrt(d))
            mp = rng.standard_normal(d)
            mq = mp - sigma * D * e
            x = mp + sigma * (u * e + zp)
            ell, Dn = V.log_ratios(x[None], mq[None], mp[None], np.array([sigma]))
            assert abs(Dn[0] - D) <= 1e-10 * D
            assert abs(ell[0] - (-u * D - 0.5 * D * D)) <= 1e-9 * max(1.0, abs(ell[0]))


def test_log_ratio_is_log_density_ratio_of_the_two_kernels():
    """ell = log N(x; m^q, s^2 I) - log N(x; m^p, s^2 I), via scipy's normal log-density."""
    rng = np.random.Generator(np.random.PCG64(12))
    B, L, d = 3, 4, 37
    x = rng.standard_normal((B, L, d)).astype(np.float32)
    mq = rng.standard_normal((B, L, d)).astype(np.float32)
    mp = (mq + 0.1 * rng.standard_normal((B, L, d))).astype(np.float32)
    s = rng.uniform(0.2, 1.5, (B, L)).astype(np.float32)
    ell, _ = V.log_ratios(x, mq, mp, s)
    x64, mq64, mp64, s64 = (a.astype(np.float64) for a in (x, mq, mp, s))
    ref = (stats.norm.logpdf(x64, mq64, s64[..., None]).sum(-1)
           - stats.norm.logpdf(x64, mp64, s64[..., None]).sum(-1))
    np.testing.assert_allclose(ell, ref, rtol=1e-10, atol=1e-10)


# ----------------------------------------------------------- sample verification
@pytest.mark.parametrize("D", [0.3, 1.0, 2.5])
def test_sample_acceptance_is_one_minus_tv(D):
    """Single-step acceptance for equal-variance Gaussians = 2 Phi(-D/2), within 3 SE of 1e6 trials."""
    n, d = 1_000_000, 4
    rng = np.random.Generator(np.random.PCG64(int(D * 1000)))
    e = _unit(rng, d)
    sigma = 0.7
    mp = np.zeros(d)
    mq = mp - sigma * D * e
    x = mp + sigma * rng.standard_normal((n, 1, d))
    ell, _ = V.log_ratios(x, mq[None, None], mp[None, None], np.full((n, 1), sigma))
    eta = philox.coins(99, np.arange(n), 1)
    tau = V.sample_verification(ell, eta, np.ones(n, dtype=np.int64))
    rate = np.mean(tau == 2)
    p = 2.0 * ndtr(-D / 2.0)
    assert abs(rate - p) < 3.0 * math.sqrt(p * (1 - p) / n)


@pytest.mark.parametrize("omega", [0.5, 2.0])
def test_tempered_sample_acceptance_matches_lemma(omega):
    """Temperature variant: P_accept(alpha=1, omega) of Lemma accept-prob."""
    n, d, D, sigma = 400_000, 3, 1.3, 0.4
    rng = np.random.Generator(np.random.PCG64(21))
    e = _unit(rng, d)
    mp = np.zeros(d)
    mq = mp - sigma * D * e
    x = mp + sigma * rng.standard_normal((n, 1, d))
    ell, _ = V.log_ratios(x, mq[None, None], mp[None, None], np.full((n, 1), sigma))
    eta = philox.coins(7, np.arange(n), 1)
    tau = V.sample_verification(ell, eta, np.ones(n, dtype=np.int64), omega=omega)
    rate = np.mean(tau == 2)
    p = accept_prob_lemma(0.0, D, omega)
    assert abs(rate - p) < 3.0 * math.sqrt(p * (1 - p) / n)


# ------------------------------------------------------------ block verification
@pytest.mark.parametrize("log_alpha,D2,omega", [(-0.7, 1.2, 1.0), (-2.5, 0.4, 1.0),
                                                (-0.3, 2.0, 1.0), (-1.0, 1.0, 1.5)])
def test_block_alpha_recursion_matches_accept_prob_lemma(log_alpha, D2, omega):
    """E[alpha_2 | alpha_1 = a] = int p min{1, a q^w/p^w} = Lemma accept-prob (L = 2)."""
    n, d, sigma = 300_000, 3, 0.5
    rng = np.random.Generator(np.random.PCG64(31))
    D1 = 0.9
    e1, e2 = _unit(rng, d), _unit(rng, d)
    mp = np.zeros((2, d))
    mq = np.stack([mp[0] - sigma * D1 * e1, mp[1] - sigma * D2 * e2])
    # step 1 fixed so that the tempered ratio gives exactly log alpha_1 = log_alpha
    u1 = (-(omega ** 2) * log_alpha - 0.5 * D1 * D1) / D1
    x = np.empty((n, 2, d))
    x[:, 0] = mp[0] + sigma * u1 * e1
    x[:, 1] = mp[1] + sigma * rng.standard_normal((n, d))
    ell, dn = V.log_ratios(x, mq[None], mp[None], np.full((n, 2), sigma))
    eta = philox.coins(3, np.arange(n), 2)
    _, _, la, _ = V.block_verification(ell, dn, eta, np.full(n, 2), omega=omega)
    np.testing.assert_allclose(la[:, 1], log_alpha, atol=1e-12)
    a2 = np.exp(la[:, 2])
    p = accept_prob_lemma(log_alpha, D2, omega)
    assert abs(a2.mean() - p) < 3.0 * a2.std() / math.sqrt(n)


@pytest.mark.parametrize("la,D", [(0.0, 0.5), (-0.1, 0.3), (-1.0, 1.0), (-3.0, 2.0),
                                  (-0.5, 4.0), (-8.0, 0.7), (-1e-4, 1e-2)])
def test_residual_mass_matches_quadrature(la, D):
    """v = alpha Phi(a+) - Phi(a-) = int max{0, alpha phi(u) - phi(u - D)} du (1-D quadrature)."""
    alpha = math.exp(la)
    f = lambda u: max(0.0, alpha * stats.norm.pdf(u) - stats.norm.pdf(u - D))
    a_plus = la / D + D / 2
    ref = integrate.quad(f, -40.0, a_plus, epsabs=0, epsrel=1e-11, limit=400)[0]
    got = math.exp(float(V.log_residual_mass(la, D)))
    assert abs(got - ref) <= 1e-8 * ref + 1e-300


def test_residual_mass_matches_2d_integral_of_kernel_difference():
    """v = int_{R^2} max{0, alpha N(z + Delta) - N(z)} dz for a 2-D Delta in a random direction."""
    rng = np.random.Generator(np.random.PCG64(41))
    for la, D in ((-0.5, 1.0), (-1.5, 0.6)):
        alpha = math.exp(la)
        th = rng.uniform(0, 2 * math.pi)
        Dx, Dy = D * math.cos(th), D * math.sin(th)
        f = lambda zy, zx: max(0.0, alpha * math.exp(-0.5 * ((zx + Dx) ** 2 + (zy + Dy) ** 2))
                               - math.exp(-0.5 * (zx * zx + zy * zy))) / (2 * math.pi)
        ref = integrate.dblquad(f, -9, 9, -9, 9, epsabs=1e-11, epsrel=1e-9)[0]
        got = math.exp(float(V.log_residual_mass(la, D)))
        assert abs(got - ref) < 2e-7


def test_block_h_limits_and_range():
    assert V.block_h(0.0, 1.0) == 1.0
    assert V.block_h(0.0, 0.0) == 1.0
    assert V.block_h(-np.inf, 1.0) == 0.0
    assert V.block_h(-0.3, 0.0) == 0.0
    la = -np.logspace(-6, 2, 60)
    for D in (0.05, 1.0, 6.0):
        h = V.block_h(la, np.full_like(la, D))
        assert np.all((h >= 0) & (h < 1))
        pos = h > 1e-300                          # h underflows for tiny alpha
        assert np.all(np.diff(h[pos]) < 0)        # smaller alpha -> smaller h
        assert np.all(np.diff(h) <= 0)
        # h = v/(v + 1 - alpha) with v from the closed form evaluated directly
        alpha = np.exp(la)
        v = alpha * ndtr(la / D + D / 2) - ndtr(la / D - D / 2)
        ok = v > 1e-12
        np.testing.assert_allclose(h[ok], (v / (v + 1 - alpha))[ok], rtol=1e-6)


def _tau_law_enumerated(p, block):
    """Exact law of tau from p_j = P(c_j = 1) by enumerating all 2^L coin patterns."""
    L = len(p)
    law = np.zeros(L + 2)
    for pattern in itertools.product([0, 1], repeat=L):
        pr = np.prod([p[j] if c else 1 - p[j] for j, c in enumerate(pattern)])
        c = [1] + list(pattern)
        if block:
            tau = 1 + max(j for j in range(L + 1) if c[j] == 1)
        else:
            fails = [j for j in range(1, L + 1) if c[j] == 0]
            tau = fails[0] if fails else L + 1
        law[tau] += pr
    return law[1:]


@pytest.mark.parametrize("block", [False, True])
def test_tau_law_matches_coin_enumeration(block):
    """For fixed (ell, D) the empirical law of tau over 2e5 coin draws matches the enumeration."""
    ell = np.array([-0.2, -1.1, 0.4, -0.6])
    dn = np.array([0.8, 1.5, 0.6, 1.1])
    L, n = 4, 200_000
    E = np.broadcast_to(ell, (n, L))
    Dm = np.broadcast_to(dn, (n, L))
    eta = philox.coins(2024, np.arange(n), L)
    g = np.full(n, L)
    if block:
        tau, _, _, h = V.block_verification(E, Dm, eta, g)
        p = h[0, 1:]
        # closed form P(tau = m+1) = h_m prod_{j>m} (1 - h_j), h_0 = 1
        hh = np.concatenate([[1.0], p])
        closed = np.array([hh[m] * np.prod(1 - hh[m + 1:]) for m in range(L + 1)])
    else:
        tau = V.sample_verification(E, eta, g)
        p = np.exp(np.minimum(0.0, ell))
        closed = np.array([np.prod(p[:t - 1]) * (1 - p[t - 1]) for t in range(1, L + 1)]
                          + [np.prod(p)])
    law = _tau_law_enumerated(p, block)
    np.testing.assert_allclose(law, closed, atol=1e-14)
    counts = np.bincount(tau, minlength=L + 2)[1:]
    pos = law > 0
    assert np.all(counts[~pos] == 0)
    assert stats.chisquare(counts[pos], law[pos] * n).pvalue > 1e-3


def _qmc_expected_tau_block(Ds, log2n=18):
    """E[tau_block] with the draft noise integrated: scrambled-Sobol quadrature over
    u_j = e_j^T Z_j ~ N(0, 1) (ell_j = -u_j D_j - D_j^2/2), coins enumerated exactly:
    P(tau = m+1 | u) = h_m prod_{j>m} (1 - h_j), h_0 = 1."""
    from scipy.stats import qmc
    from scipy.special import ndtri
    L = len(Ds)
    pts = qmc.Sobol(d=L, scramble=True, seed=1234).random_base2(log2n)
    U = ndtri(pts)
    Ds = np.asarray(Ds)
    ell = -U * Ds - 0.5 * Ds * Ds
    n = U.shape[0]
    _, _, _, h = V.block_verification(ell, np.broadcast_to(Ds, (n, L)), np.ones((n, L)),
                                      np.full(n, L))
    hh = h.copy()
    hh[:, 0] = 1.0
    et = np.zeros(n)
    for m in range(L + 1):
        et += (m + 1) * hh[:, m] * np.prod(1 - hh[:, m + 1:], axis=1)
    return float(et.mean())


@pytest.mark.parametrize("Ds", [(0.7,), (0.5, 1.4), (1.2, 0.3, 0.9)])
def test_expected_tau_brute_force_small_d(Ds):
    """E[tau] over drafts and coins at d <= 4, L <= 3: oracle Monte Carlo vs closed form / quadrature."""
    L, d, n, sigma = len(Ds), 4, 200_000, 0.8
    rng = np.random.Generator(np.random.PCG64(51 + L))
    es = np.stack([_unit(rng, d) for _ in range(L)])
    mp = rng.standard_normal((L, d))
    mq = mp - sigma * np.asarray(Ds)[:, None] * es
    x = mp + sigma * rng.standard_normal((n, L, d))
    ell, dn = V.log_ratios(x, mq[None], mp[None], np.full((n, L), sigma))
    eta = philox.coins(17, np.arange(n), L)
    g = np.full(n, L)
    t_s = V.sample_verification(ell, eta, g)
    t_b = V.block_verification(ell, dn, eta, g)[0]
    a = 2.0 * ndtr(-np.asarray(Ds) / 2.0)
    e_sample = sum(np.prod(a[:t]) for t in range(L + 1))
    e_block = _qmc_expected_tau_block(Ds)
    assert abs(t_s.mean() - e_sample) < 3 * t_s.std() / math.sqrt(n)
    assert abs(t_b.mean() - e_block) < 3 * t_b.std() / math.sqrt(n)
    assert e_block >= e_sample - 1e-4          # block is never worse in expectation
    if L == 1:
        assert abs(e_block - e_sample) < 1e-4    # h_1 = alpha_1: the two rules coincide


def test_block_equals_sample_when_L_is_one():
    rng = np.random.Generator(np.random.PCG64(61))
    n = 5000
    ell = rng.normal(-0.5, 1.0, (n, 1))
    dn = rng.uniform(0.1, 3, (n, 1))
    eta = philox.coins(5, np.arange(n), 1)
    g = np.ones(n, dtype=np.int64)
    np.testing.assert_array_equal(V.sample_verification(ell, eta, g),
                                  V.block_verification(ell, dn, eta, g)[0])


def test_equal_means_accept_everything():
    rng = np.random.Generator(np.random.PCG64(62))
    B, L, d = 6, 5, 9
    mp = rng.standard_normal((B, L, d))
    x = rng.standard_normal((B, L, d))
    for mode in (V.MODE_SAMPLE, V.MODE_BLOCK):
        r = V.verify(x, mp, mp, np.ones((B, L)), 3, mode)
        assert np.all(r["tau"] == L + 1)
        np.testing.assert_array_equal(r["y"], x[:, -1])


# ------------------------------------------------------------------ residual
@pytest.mark.parametrize("la,D", [(0.0, 1.0), (-0.8, 0.5), (-3.0, 2.5), (0.0, 0.05), (-12.0, 1.0)])
def test_psi_cdf_matches_quadrature(la, D):
    alpha = math.exp(la)
    f = lambda u: max(0.0, alpha * stats.norm.pdf(u) - stats.norm.pdf(u - D))
    a_plus = la / D + D / 2
    total = integrate.quad(f, a_plus - 40.0, a_plus, epsabs=0, epsrel=1e-12, limit=400)[0]
    for q in (0.02, 0.3, 0.5, 0.9, 0.999):
        u = a_plus - q * 6.0 / (1.0 + abs(a_plus) + D)
        ref = integrate.quad(f, a_plus - 40.0, u, epsabs=0, epsrel=1e-12, limit=400)[0] / total
        assert abs(float(V.psi_cdf(u, D, la)) - ref) < 1e-8
    assert float(V.psi_cdf(a_plus, D, la)) == 1.0
    assert float(V.psi_cdf(a_plus + 1.0, D, la)) == 1.0
    # at the upper bound the two scaled densities cross: alpha phi(a+) = phi(a-)
    assert math.isclose(alpha * stats.norm.pdf(a_plus), stats.norm.pdf(a_plus - D), rel_tol=1e-9)


def test_usample_inverts_psi():
    rng = np.random.Generator(np.random.PCG64(71))
    n = 3000
    D = rng.uniform(0.01, 6.0, n)
    la = -rng.exponential(1.5, n) * (rng.uniform(size=n) < 0.7)
    w = philox.uniform_of(rng.integers(0, 2 ** 32, n))
    U = V.usample_bisection(D, la, w)
    a_plus = la / D + D / 2
    assert np.all(U <= a_plus)
    np.testing.assert_allclose(V.psi_cdf(U, D, la), w, atol=1e-9)
    # extreme uniforms from the 32-bit words 0 and 2^32 - 1
    for word in (0, 1, 2 ** 31, 2 ** 32 - 2, 2 ** 32 - 1):
        wv = float(philox.uniform_of(word))
        Ux = V.usample_bisection(np.array([1.3]), np.array([-0.4]), np.array([wv]))
        assert abs(float(V.psi_cdf(Ux, 1.3, -0.4)[0]) - wv) < 1e-9


@pytest.mark.parametrize("D", [0.4, 1.0, 3.0])
def test_residual_mean_at_alpha_one(D):
    """e^T(Y - m^q)/sigma has mean -D (1 - Phi(D/2)) / (2 Phi(D/2) - 1) when alpha = 1."""
    n = 200_000
    w = philox.usample_uniform(88, np.arange(n))
    U = V.usample_bisection(np.full(n, D), np.zeros(n), w)
    ref = -D * (1.0 - ndtr(D / 2)) / (2.0 * ndtr(D / 2) - 1.0)
    assert abs(U.mean() - ref) < 3 * U.std() / math.sqrt(n)
    assert stats.kstest(U, lambda u: V.psi_cdf(u, np.full(np.shape(u), D),
                                               np.zeros(np.shape(u)))).pvalue > 1e-3


def test_residual_perpendicular_part_moments():
    rng = np.random.Generator(np.random.PCG64(81))
    d, n = 3, 200_000
    Delta = 1.7 * _unit(rng, d)
    e = Delta / np.linalg.norm(Delta)
    G = philox.normals(9, np.arange(n), d, philox.STREAM_RESID)
    U = np.full(n, 0.25)
    Y = V.decomposition_residual(np.broadcast_to(Delta, (n, d)), np.zeros((n, d)),
                                 np.ones(n), U, G)
    np.testing.assert_allclose(Y @ e, 0.25, atol=1e-12)
    Zp = Y - 0.25 * e
    assert np.all(np.abs(Zp.mean(0)) < 5 / math.sqrt(n))
    cov = np.cov(Zp.T)
    assert np.max(np.abs(cov - (np.eye(d) - np.outer(e, e)))) < 0.02


def _fixed_mean_window(rng, L, d, Ds, sigma):
    es = np.stack([_unit(rng, d) for _ in range(L)])
    mp = rng.standard_normal((L, d))
    mq = mp - sigma * np.asarray(Ds)[:, None] * es
    return es, mp, mq


@pytest.mark.parametrize("mode,residual", [(V.MODE_SAMPLE, V.RESIDUAL_DECOMPOSITION),
                                           (V.MODE_BLOCK, V.RESIDUAL_DECOMPOSITION),
                                           (V.MODE_SAMPLE, V.RESIDUAL_REFLECTION)])
def test_single_step_output_follows_target(mode, residual):
    """L = 1: the emitted state (accepted draft or residual) is exactly N(m^q, sigma^2 I)."""
    rng = np.random.Generator(np.random.PCG64(91))
    n, d, sigma = 60_000, 3, 0.6
    e, mp, mq = _fixed_mean_window(rng, 1, d, [1.1], sigma)
    x = mp[None] + sigma * rng.standard_normal((n, 1, d))
    r = V.verify(x, np.broadcast_to(mq, (n, 1, d)), np.broadcast_to(mp, (n, 1, d)),
                 np.full((n, 1), sigma), 4242, mode, residual=residual)
    y = np.where((r["tau"] == 2)[:, None], x[:, 0], r["y"])
    z = (y - mq[0]) / sigma
    assert stats.kstest(z @ e[0], "norm").pvalue > 1e-3
    perp = _perp(rng, e[0])
    assert stats.kstest(z @ perp, "norm").pvalue > 1e-3
    assert np.max(np.abs(np.cov(z.T) - np.eye(d))) < 0.03


def test_block_two_step_output_follows_target():
    """L = 2 block verification + continuation from q: (Y_1, Y_2) ~ q_1 x q_2 (fixed means)."""
    rng = np.random.Generator(np.random.PCG64(92))
    n, d, sigma = 80_000, 3, 0.5
    es, mp, mq = _fixed_mean_window(rng, 2, d, [1.0, 1.6], sigma)
    x = mp[None] + sigma * rng.standard_normal((n, 2, d))
    r = V.verify(x, np.broadcast_to(mq, (n, 2, d)), np.broadcast_to(mp, (n, 2, d)),
                 np.full((n, 2), sigma), 777, V.MODE_BLOCK)
    tau = r["tau"]
    assert np.any(tau == 1) and np.any(tau == 2) and np.any(tau == 3)
    assert np.any(r["log_alpha_res"][tau == 2] < 0)       # residual with alpha_res < 1 exercised
    fresh = mq[1] + sigma * rng.standard_normal((n, d))
    Y1 = np.where((tau == 1)[:, None], r["y"], x[:, 0])
    Y2 = np.where((tau == 1)[:, None], fresh, np.where((tau == 2)[:, None], r["y"], x[:, 1]))
    z1 = (Y1 - mq[0]) / sigma @ es[0]
    z2 = (Y2 - mq[1]) / sigma @ es[1]
    assert stats.kstest(z1, "norm").pvalue > 1e-3
    assert stats.kstest(z2, "norm").pvalue > 1e-3
    assert abs(np.corrcoef(z1, z2)[0, 1]) < 4 / math.sqrt(n)


def test_verify_ragged_windows_and_bonus():
    """Leff < L uses only the first Leff steps; a full accept takes the bonus step when given."""
    rng = np.random.Generator(np.random.PCG64(93))
    B, L, d = 8, 5, 6
    mp = rng.standard_normal((B, L, d))
    x = rng.standard_normal((B, L, d))
    Leff = np.array([1, 2, 3, 5, 5, 4, 2, 1])
    mqb = rng.standard_normal((B, d))
    sb = rng.uniform(0.1, 1, B)
    r = V.verify(x, mp, mp, np.ones((B, L)), 9, V.MODE_BLOCK, Leff=Leff,
                 mu_target_bonus=mqb, sigma_bonus=sb)
    assert np.all(r["tau"] == Leff + 1)
    Gb = philox.normals(9, np.arange(B), d, philox.STREAM_BONUS)
    np.testing.assert_allclose(r["y"], mqb + sb[:, None] * Gb, rtol=1e-14)
    # steps past Leff never influence the result
    x2 = x.copy()
    mq = mp.copy()
    mq[:, :, 0] += 0.7
    mq2 = mq.copy()
    for b in range(B):
        x2[b, Leff[b]:] = 1e6
        mq2[b, Leff[b]:] = -1e6
    r1 = V.verify(x, mq, mp, np.ones((B, L)), 9, V.MODE_BLOCK, Leff=Leff)
    r2 = V.verify(x2, mq2, mp, np.ones((B, L)), 9, V.MODE_BLOCK, Leff=Leff)
    np.testing.assert_array_equal(r1["tau"], r2["tau"])
    np.testing.assert_array_equal(r1["y"], r2["y"])
