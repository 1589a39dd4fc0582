"""Pins for the fp64 sampler oracle: the VP schedule, the GMM score, the Euler-Maruyama
chain and the speculative samplers (Free / Frozen drafter, sample / block verification).

Independent references: quadrature of beta, finite differences of the mixture
log-density (scipy), the closed-form law of the linear (one-component) chain, the
paper's remark that the Frozen drafter's first draft is always accepted, and the data
law itself: for Gaussian data the reverse chain must reach N(mu, s^2 I) at first order
in 1/K for every churn (this pins the drift and the noise scale of the target mean
against the forward process alone; planted misreadings of either fail it).
"""
import math

import numpy as np
import pytest
from scipy import integrate, stats
from scipy.special import logsumexp

from oracle import sampler as S
from oracle import verify as V


def _gmm(C, d, seed, comp_var=1.0, scale=2.0):
    rng = np.random.Generator(np.random.PCG64(seed))
    means = scale * rng.standard_normal((C, d))
    w = rng.dirichlet(np.ones(C))
    return dict(means=means, log_weights=np.log(w), comp_var=comp_var)


def test_alpha_bar_is_exp_of_integrated_beta():
    sch = S.VPSchedule(K=100, churn=0.5)
    for t in (1e-4, 0.1, 0.5, 0.93, 1.0):
        ref = math.exp(-integrate.quad(lambda s: float(sch.beta(s)), 0, t)[0])
        assert abs(float(sch.alpha_bar(t)) - ref) < 1e-12
    # sigma_k = sqrt(delta) * churn * g_{1 - t_k}, g = sqrt(beta)
    assert abs(float(sch.sigma(10)) - math.sqrt(0.01) * 0.5 * math.sqrt(float(sch.beta(0.9)))) < 1e-15
    assert float(sch.tfwd(100)) == 1e-4


def test_gmm_score_is_gradient_of_log_density():
    sch = S.VPSchedule(K=100, churn=0.5)
    gmm = _gmm(5, 4, 1)
    rng = np.random.Generator(np.random.PCG64(2))

    def logq(x, tf):
        ab = float(sch.alpha_bar(tf))
        v = ab * gmm["comp_var"] + 1 - ab
        comps = [lw + stats.multivariate_normal.logpdf(x, math.sqrt(ab) * mu, v * np.eye(4))
                 for lw, mu in zip(gmm["log_weights"], gmm["means"])]
        return logsumexp(comps)

    for tf in (0.02, 0.3, 0.9):
        for _ in range(4):
            x = 2.5 * rng.standard_normal(4)
            s = S.gmm_score(x[None], np.array([tf]), gmm["means"], gmm["log_weights"],
                            gmm["comp_var"], sch)[0]
            h = 1e-5
            fd = np.array([(logq(x + h * e, tf) - logq(x - h * e, tf)) / (2 * h) for e in np.eye(4)])
            np.testing.assert_allclose(s, fd, rtol=1e-5, atol=1e-6)


def _check_law(y, m, var, n_sigma=4.0):
    n, d = y.shape
    se_m = math.sqrt(var / n)
    assert np.all(np.abs(y.mean(0) - m) < n_sigma * se_m), (y.mean(0), m)
    se_v = var * math.sqrt(2.0 / (n - 1))
    assert np.all(np.abs(y.var(0) - var) < n_sigma * se_v), (y.var(0), var)
    for c in range(d):
        assert stats.kstest((y[:, c] - m[c]) / math.sqrt(var), "norm").pvalue > 1e-3


@pytest.fixture(scope="module", params=[40, 3])
def linear_setup(request):
    """K = 40 (many rounds) and K = 3 < L (a single window that reaches the end of
    sampling, where a full accept must stop at yhat_K and take no bonus step)."""
    sch = S.VPSchedule(K=request.param, churn=0.8)
    gmm = dict(means=np.array([[1.5, -2.0, 0.5]]), log_weights=np.zeros(1), comp_var=0.5)
    m, var = S.linear_gaussian_moments(gmm["means"][0], gmm["comp_var"], sch)
    return sch, gmm, m, var


def test_em_chain_matches_linear_closed_form(linear_setup):
    sch, gmm, m, var = linear_setup
    y = S.em_sample(20000, 3, gmm, sch, seed=3)
    _check_law(y, m, var)


@pytest.mark.parametrize("mode,drafter", [(V.MODE_SAMPLE, "free"), (V.MODE_BLOCK, "free"),
                                          (V.MODE_BLOCK, "frozen")])
def test_speculative_sampler_matches_linear_closed_form(linear_setup, mode, drafter):
    """Exactness of the whole round (drafter, verification, residual, bonus, end handling,
    score cache): Y_K has the law of the plain EM chain."""
    sch, gmm, m, var = linear_setup
    out = S.speculative_sample(20000, 3, 4, mode, gmm, sch, seed=4, drafter=drafter)
    assert np.all(out["k"] == sch.K)
    _check_law(out["y"], m, var)
    assert 1 <= out["rounds"] <= sch.K


def test_frozen_drafter_always_accepts_its_first_draft():
    sch = S.VPSchedule(K=30, churn=0.5)
    gmm = _gmm(3, 4, 5)
    out = S.speculative_sample(300, 4, 4, V.MODE_SAMPLE, gmm, sch, seed=6, drafter="frozen")
    for t in out["taus"]:
        assert np.all((t == 0) | (t >= 2))


def test_block_is_more_efficient_than_sample_on_the_mixture():
    sch = S.VPSchedule(K=60, churn=0.5)
    gmm = _gmm(4, 6, 7)
    r = {m: S.speculative_sample(400, 6, 6, m, gmm, sch, seed=8) for m in (0, 1)}
    # fewer rounds (parallel target calls) per chain with block verification
    assert r[1]["chain_rounds"].mean() < r[0]["chain_rounds"].mean()
    for m in (0, 1):
        assert np.all(r[m]["k"] == sch.K)
        taus = np.concatenate([t[t > 0] for t in r[m]["taus"]])
        # every chain covers K steps: the taus of a chain sum to at least K
        assert taus.sum() >= 400 * sch.K


def test_speculative_and_em_agree_on_the_mixture():
    """Two-sample checks between the speculative samplers and the plain chain (8 components)."""
    sch = S.VPSchedule(K=50, churn=0.5)
    gmm = _gmm(8, 4, 9)
    n = 4000
    y_em = S.em_sample(n, 4, gmm, sch, seed=10)
    rng = np.random.Generator(np.random.PCG64(11))
    dirs = rng.standard_normal((3, 4))
    for mode in (V.MODE_SAMPLE, V.MODE_BLOCK):
        y_sp = S.speculative_sample(n, 4, 5, mode, gmm, sch, seed=12)["y"]
        for u in dirs:
            assert stats.ks_2samp(y_em @ u, y_sp @ u).pvalue > 1e-3


# ---- the reverse-SDE drift against the data law (Eq. forward-process, Eq. backward-process)
#
# For Gaussian data N(mu, s^2 I) the forward process has the closed-form marginals
# q_t = N(sqrt(abar_t) mu, (abar_t s^2 + 1 - abar_t) I).  For every churn eps, the
# reverse SDE with drift -f y + (1 + eps^2)/2 g^2 score and diffusion eps g, started
# from q_1, has the marginals q_{1-t}; at the end of sampling that is the data law
# itself.  The oracle's Euler-Maruyama chain must therefore reach N(mu, s^2 I) with
# an error of first order in delta = 1/K.  With one component the oracle's target
# mean is affine in y, so the law of Y_K is propagated exactly (mean and covariance)
# through target_mean and VPSchedule.sigma as they stand; the only inputs that do not
# come from the oracle's reverse-time code are q_1 (the forward closed form) and the
# data law.  The forward-time floor (1e-4) touches only the last steps of K = 1e5 and
# its bias is below the first-order error there.

def _propagate_law(K, churn, mu, s2, target_mean=S.target_mean, sigma=None):
    sch = S.VPSchedule(K=K, churn=churn)
    gmm = dict(means=np.asarray(mu, np.float64)[None], log_weights=np.zeros(1), comp_var=s2)
    d = len(mu)
    ab1 = float(sch.alpha_bar(1.0))
    m = math.sqrt(ab1) * np.asarray(mu, np.float64)
    P = (ab1 * s2 + 1.0 - ab1) * np.eye(d)
    basis = np.vstack([np.zeros(d), np.eye(d)])      # y = 0 and the unit vectors
    for k in range(K):
        out, _ = target_mean(basis, np.full(d + 1, k), gmm, sch)
        c = out[0]
        A = (out[1:] - c).T                           # m^q_k(y) = A y + c
        sk = float(sch.sigma(k)) if sigma is None else sigma(sch, k)
        m = A @ m + c
        P = A @ P @ A.T + sk * sk * np.eye(d)
    return m, P


def _law_error(m, P, mu, s2):
    return (np.abs(m - mu).max(), np.abs(np.diag(P) - s2).max(),
            np.abs(P - np.diag(np.diag(P))).max())


_MU = np.array([1.5, -2.0, 0.5])


@pytest.mark.parametrize("s2", [0.5, 2.0])
@pytest.mark.parametrize("churn", [0.0, 0.5, 1.5])
def test_reverse_chain_reaches_the_data_law(s2, churn):
    errs = []
    for K in (1000, 10000):
        em, ev, eo = _law_error(*_propagate_law(K, churn, _MU, s2), _MU, s2)
        assert eo < 1e-12
        assert max(em, ev) < 4.0 / K, (K, em, ev)
        errs.append(max(em, ev))
    # first order in delta: ten times more steps, ten times less error
    assert 8.0 < errs[0] / errs[1] < 12.5, errs


def test_reverse_chain_reaches_the_data_law_at_1e5_steps():
    em, ev, _ = _law_error(*_propagate_law(100000, 0.5, _MU, 0.5), _MU, 0.5)
    assert max(em, ev) < 4e-5, (em, ev)


def _planted_flipped_f(y, k, gmm, sched):
    """target_mean with the sign of f reversed (a planted mistake)."""
    y = np.asarray(y, np.float64)
    tf = sched.tfwd(k)
    b = np.broadcast_to(sched.beta(tf), y.shape[:-1])[..., None]
    s = S.gmm_score(y, tf, gmm["means"], gmm["log_weights"], gmm["comp_var"], sched)
    return y + sched.delta * (-0.5 * b * y + 0.5 * (1.0 + sched.churn ** 2) * b * s), s


def _planted_no_churn_factor(y, k, gmm, sched):
    """target_mean without the (1 + eps^2)/2 factor on the score term (a planted mistake)."""
    y = np.asarray(y, np.float64)
    tf = sched.tfwd(k)
    b = np.broadcast_to(sched.beta(tf), y.shape[:-1])[..., None]
    s = S.gmm_score(y, tf, gmm["means"], gmm["log_weights"], gmm["comp_var"], sched)
    return y + sched.delta * (0.5 * b * y + b * s), s


def _planted_sigma_without_sqrt_delta(sched, k):
    return sched.churn * math.sqrt(float(sched.beta(sched.tfwd(k))))


@pytest.mark.parametrize("churn", [0.5, 1.5])
def test_drift_pin_catches_planted_mistakes(churn):
    """The pin above fails, by far, for each plausible misreading of the drift or noise."""
    K, s2 = 10000, 0.5
    for kw in (dict(target_mean=_planted_flipped_f), dict(target_mean=_planted_no_churn_factor),
               dict(sigma=_planted_sigma_without_sqrt_delta)):
        em, ev, _ = _law_error(*_propagate_law(K, churn, _MU, s2, **kw), _MU, s2)
        assert max(em, ev) > 0.1, kw


@pytest.mark.parametrize("mode,drafter", [(V.MODE_SAMPLE, "free"), (V.MODE_BLOCK, "frozen")])
def test_chain_subset_equals_rows_of_the_full_run(mode, drafter):
    """Random numbers are keyed by chain index, so sampling a subset of the chains (as the
    GPU parity tests do at full batch size) gives exactly those rows of the full run."""
    sch = S.VPSchedule(K=25, churn=0.5)
    gmm = _gmm(3, 5, 13)
    full = S.speculative_sample(12, 5, 4, mode, gmm, sch, seed=14, drafter=drafter,
                                return_trace=True)
    sub = np.array([1, 4, 5, 11])
    part = S.speculative_sample(12, 5, 4, mode, gmm, sch, seed=14, drafter=drafter, chains=sub,
                                return_trace=True)
    np.testing.assert_array_equal(part["y"], full["y"][sub])
    np.testing.assert_array_equal(part["k"], full["k"][sub])
    for tp, tf in zip(part["trace"], full["trace"]):
        np.testing.assert_array_equal(tp["tau"], tf["tau"][sub])
