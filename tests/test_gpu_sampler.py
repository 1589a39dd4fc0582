"""GPU parity of the end-to-end sampler pieces (C ABI, sm_103a) against the fp64 oracle:
the Gaussian-mixture target call, the drafter, the plain Euler-Maruyama chain, the first
rounds of the speculative sampler element by element, and the law of Y_K."""
import math

import numpy as np
import pytest
import torch
from scipy import stats

import workloads as W
from oracle import sampler as OS
from oracle import verify as OV
from gpu_helpers import near_tie

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def api():
    import __graft_entry__ as g
    g.build()
    from paper_2606_13426_gb300 import api as A
    return A


def _gmm(C, d, seed, comp_var=1.0):
    rng = np.random.Generator(np.random.PCG64(seed))
    means = (2.0 * rng.standard_normal((C, d))).astype(np.float32)
    lw = np.log(rng.dirichlet(np.ones(C))).astype(np.float32)
    return dict(means=means, log_weights=lw, comp_var=comp_var)


def _target(api, gmm, K, churn):
    return api.GmmTarget(torch.from_numpy(gmm["means"]), torch.from_numpy(gmm["log_weights"]),
                         gmm["comp_var"], K, churn)


def _score_error_bound(z, k, gmm, sch, gamma=32 * 2.0 ** -24):
    """Per-element bound on the fp32 error of the mixture score at rows z (fp64 inputs).

    The logits are log w_c - D_c / (2 v) with D_c = |z - sqrt(abar) mu_c|^2 summed in fp32,
    whose relative error is at most gamma (a few ulps per level of the reduction; 32 ulps
    covers any order the kernels use for d <= 4096).  A logit error e_c moves the
    responsibilities by dr_c = r_c (e_c - sum_b r_b e_b), and the score by
    sum_c dr_c sqrt(abar) mu_c / v, so |ds_i| <= 2 max_c |e_c| sum_c r_c |sqrt(abar) mu_ci - sbar_i| / v
    with sbar = sum_c r_c sqrt(abar) mu_c.  Where one component dominates the sum is tiny;
    two comparable components far from z are the worst case.  Plain rounding of the final
    combination adds a few ulps of |z|/v and |sqrt(abar) mu|/v."""
    tf = sch.tfwd(k)
    ab = sch.alpha_bar(tf)
    v = ab * gmm["comp_var"] + 1.0 - ab
    cen = np.sqrt(ab)[:, None, None] * gmm["means"].astype(np.float64)[None]     # [n, C, d]
    D = np.sum((z[:, None, :] - cen) ** 2, axis=-1)                             # [n, C]
    lg = gmm["log_weights"].astype(np.float64)[None] - D / (2.0 * v[:, None])
    r = np.exp(lg - lg.max(axis=1, keepdims=True))
    r /= r.sum(axis=1, keepdims=True)
    e = gamma * D / (2.0 * v[:, None]) + 2.0 ** -23 * np.abs(lg)
    emax = np.max(np.where(r > 1e-30, e, 0.0), axis=1)
    sbar = np.sum(r[:, :, None] * cen, axis=1)
    dev = np.sum(r[:, :, None] * np.abs(cen - sbar[:, None, :]), axis=1)
    mag = (np.abs(z) + np.abs(cen).max(axis=1)) / v[:, None]
    return 2.0 * emax[:, None] * dev / v[:, None] + 8 * 2.0 ** -24 * mag


@pytest.mark.parametrize("d", [1024, 37])
def test_gmm_target_matches_oracle(api, d):
    """The target call (Eq. target-distribution with the mixture score): on states near the
    noised mixture at their own step the mean is within the output-state tolerance (1e-5
    absolute); on every state the score is within the fp32 error bound of the softmax
    over the squared distances (_score_error_bound), which also bounds the mean through
    the factor delta (1 + eps^2)/2 beta."""
    gmm = _gmm(8, d, 1)
    K = 1000
    sch = OS.VPSchedule(K, 0.5)
    rng = np.random.Generator(np.random.PCG64(2))
    n = 192
    k = rng.integers(0, K + 1, n).astype(np.int32)
    tf = sch.tfwd(k)
    ab = sch.alpha_bar(tf)
    comp = rng.integers(0, 8, n)
    z = (np.sqrt(ab)[:, None] * gmm["means"][comp]
         + np.sqrt(ab * gmm["comp_var"] + 1 - ab)[:, None] * rng.standard_normal((n, d)))
    generic = np.zeros(n, dtype=bool)
    generic[::7] = True                       # generic points far from every component
    z[generic] = 3.0 * rng.standard_normal((int(generic.sum()), d))
    z = z.astype(np.float32)
    mq, sc = api.gmm_target(torch.from_numpy(z).cuda(), torch.from_numpy(k).cuda(),
                            _target(api, gmm, K, 0.5))
    mq, sc = mq.cpu().numpy(), sc.cpu().numpy()
    z64 = z.astype(np.float64)
    mq_o, sc_o = OS.target_mean(z64, k, gmm, sch)
    bound = _score_error_bound(z64, k, gmm, sch)
    err_s = np.abs(sc - sc_o)
    assert np.all(err_s <= bound), "score error above its fp32 bound: %g" % np.max(err_s / bound)
    b = sch.beta(tf)[:, None]
    mbound = sch.delta * 0.5 * (1 + 0.25) * b * bound + 4 * 2.0 ** -24 * (np.abs(mq_o) + np.abs(z64))
    err_m = np.abs(mq - mq_o)
    assert np.all(err_m <= mbound + 1e-7)
    assert err_m[~generic].max() <= 1e-5, err_m[~generic].max()
    print("target call d=%d: mean err %.3g (on-manifold %.3g), score err %.3g, worst err/bound %.3g"
          % (d, err_m.max(), err_m[~generic].max(), err_s.max(), np.max(err_s / bound)))


def test_free_draft_matches_oracle(api):
    d, Bn, L, K = 300, 40, 6, 200
    sch = OS.VPSchedule(K, 0.7)
    rng = np.random.Generator(np.random.PCG64(3))
    y = rng.standard_normal((Bn, d)).astype(np.float32)
    s = rng.standard_normal((Bn, d)).astype(np.float32)
    k = rng.integers(0, K, Bn).astype(np.int32)
    g = np.minimum(rng.integers(0, L + 1, Bn), K - k).astype(np.int32)
    tgt = _target(api, _gmm(2, d, 4), K, 0.7)
    x, mp, sg = api.free_draft(torch.from_numpy(y).cuda(), torch.from_numpy(s).cuda(),
                               torch.from_numpy(k).cuda(), torch.from_numpy(g).cuda(), L, tgt, 77)
    x, mp, sg = x.cpu().numpy(), mp.cpu().numpy(), sg.cpu().numpy()
    xo, mpo, sgo = OS.draft(y.astype(np.float64), s.astype(np.float64), k.astype(np.int64), g, L,
                            sch, 77, np.arange(Bn))
    live = np.arange(L)[None, :] < g[:, None]
    print("drafter: max |x - x_oracle| %.3g, max |m^p - m^p_oracle| %.3g"
          % (np.abs(x - xo)[live].max(), np.abs(mp - mpo)[live].max()))
    assert np.max(np.abs(x - xo)[live]) <= 1e-5
    assert np.max(np.abs(mp - mpo)[live]) <= 1e-5
    assert np.max(np.abs(sg - sgo)[live] / sgo[live]) < 1e-6


@pytest.mark.parametrize("K,Bn,d,chains", [(12, 32, 64, None), (1000, 1024, 1024, 24)])
def test_em_chain_matches_oracle(api, K, Bn, d, chains):
    """The plain Euler-Maruyama chain: a few very long steps, and the sampler workload's
    schedule (K = 1000, B = 1024, d = 1024, 8 components; 24 chains followed by the
    oracle).  Each fp32 step y + delta b(y) + sigma G rounds the state by a few ulps and
    the chain's Jacobian stays close to 1, so the rounding performs a random walk over
    the K steps: the tolerance is the output-state tolerance (1e-5 absolute) for short
    chains and 4 sqrt(K) * 2 ulps of the largest state beyond that."""
    gmm = _gmm(8, d, 5)
    sch = OS.VPSchedule(K, 0.5)
    ch = np.arange(Bn) if chains is None else np.linspace(0, Bn - 1, chains).astype(int)
    y = api.em_sample(Bn, _target(api, gmm, K, 0.5), 9).cpu().numpy()[ch]
    yo = OS.em_sample(Bn, d, gmm, sch, 9, chains=ch)
    err = np.abs(y - yo).max()
    tol = max(1e-5, 4.0 * math.sqrt(K) * 2.0 * 2.0 ** -24 * np.abs(yo).max())
    print("EM chain K=%d d=%d: max |y - y_oracle| %.3g (tolerance %.3g)" % (K, d, err, tol))
    assert err <= tol


def _first_rounds(api, mode, drafter, d, C, Bn=192, L=4, K=40, gmm=None, chains=None, churn=0.5,
                  seed=123):
    """Rounds 1..3 of the GPU sampler (all Bn chains) against the oracle on `chains`: k
    bit-exact and the emitted states within the output-state tolerance (1e-5 absolute,
    fp32) for the chains whose coins lie outside the tie band in every round so far."""
    gmm = _gmm(C, d, 6) if gmm is None else gmm
    sch = OS.VPSchedule(K, churn)
    tgt = _target(api, gmm, K, churn)
    chains = np.arange(Bn) if chains is None else np.asarray(chains)
    o = OS.speculative_sample(Bn, d, L, mode, gmm, sch, seed=seed, drafter=drafter, max_rounds=3,
                              chains=chains, return_trace=True)
    clean = np.ones(len(chains), dtype=bool)
    worst = 0.0
    for R in (1, 2, 3):
        r = api.sampler_run(Bn, L, tgt, seed, "block" if mode else "sample", drafter, max_rounds=R)
        assert r["rounds"] == R
        tr = o["trace"][R - 1]
        clean &= ~near_tie(tr["res"], mode)
        k = r["k"].cpu().numpy()[chains]
        y = r["y"].cpu().numpy()[chains]
        assert clean.mean() > 0.9
        np.testing.assert_array_equal(k[clean], tr["k"][clean])
        err = np.abs(y[clean] - tr["y"][clean])
        worst = max(worst, float(err.max()))
        assert err.max() <= 1e-5, (R, err.max())
    return worst


@pytest.mark.parametrize("mode", [OV.MODE_SAMPLE, OV.MODE_BLOCK])
@pytest.mark.parametrize("drafter", ["free", "frozen"])
def test_first_rounds_match_oracle(api, mode, drafter):
    """Rounds 1..3 element by element: k, and the states of chains whose coins all lie
    outside the tie band in every round so far."""
    _first_rounds(api, mode, drafter, 64, 8)


@pytest.mark.parametrize("L", [4, 8, 16])
@pytest.mark.parametrize("mode", [OV.MODE_SAMPLE, OV.MODE_BLOCK])
@pytest.mark.parametrize("drafter", ["free", "frozen"])
def test_first_rounds_match_oracle_at_sampler_workload_shape(api, L, mode, drafter):
    """The end-to-end sampler workload itself: 8-component mixture in d = 1024, K = 1000
    VP steps, B = 1024 chains (the verification takes its many-chain path), windows
    L in {4, 8, 16}; 40 chains spread over the batch are followed by the oracle."""
    cfg = W.SAMPLER_CONFIG
    chains = np.unique(np.concatenate([np.linspace(0, cfg["B"] - 1, 39).astype(int), [cfg["B"] - 1]]))
    worst = _first_rounds(api, mode, drafter, cfg["d"], cfg["n_components"], Bn=cfg["B"], L=L,
                          K=cfg["K"], gmm=W.make_gmm(), chains=chains, churn=cfg["churn"])
    print("sampler workload L=%d mode=%d %s: max |y - y_oracle| %.3g" % (L, mode, drafter, worst))


@pytest.mark.parametrize("mode,drafter", [("block", "free"), ("sample", "frozen")])
def test_host_driven_rounds_equal_graph_run(api, mode, drafter):
    """begin + R rounds + end launches the kernels of R iterations of the round graph:
    identical outputs, bit for bit."""
    d, Bn, L, K = 64, 160, 4, 40
    tgt = _target(api, _gmm(8, d, 11), K, 0.5)
    for R in (1, 5):
        g = api.sampler_run(Bn, L, tgt, 77, mode, drafter, max_rounds=R)
        h = api.sampler_rounds(Bn, L, tgt, 77, R, mode, drafter)
        assert g["rounds"] == h["rounds"] == R
        for key in ("y", "k", "chain_rounds", "tau_sum"):
            assert torch.equal(g[key], h[key]), key


# Row lengths and component counts that take the other target-call kernels: ragged d
# and rows longer than 1024 elements (shared-memory means), 9..16 components.
@pytest.mark.parametrize("d,C", [(37, 8), (1100, 8), (64, 12), (1024, 12), (1030, 12)])
def test_first_rounds_other_shapes(api, d, C):
    _first_rounds(api, OV.MODE_BLOCK, "free", d, C, Bn=96)


def _check_law(y, m, var, n_sigma=4.0):
    n = y.shape[0]
    assert np.all(np.abs(y.mean(0) - m) < n_sigma * math.sqrt(var / n))
    assert np.all(np.abs(y.var(0) - var) < n_sigma * var * math.sqrt(2.0 / (n - 1)))
    for c in range(y.shape[1]):
        assert stats.kstest((y[:, c] - m[c]) / math.sqrt(var), "norm").pvalue > 1e-3


@pytest.mark.parametrize("K", [40, 3])
@pytest.mark.parametrize("mode,drafter", [("sample", "free"), ("block", "free"),
                                          ("block", "frozen")])
def test_gpu_sampler_matches_linear_closed_form(api, K, mode, drafter):
    gmm = dict(means=np.array([[1.5, -2.0, 0.5]], np.float32), log_weights=np.zeros(1, np.float32),
               comp_var=0.5)
    sch = OS.VPSchedule(K, 0.8)
    m, var = OS.linear_gaussian_moments(gmm["means"][0].astype(np.float64), 0.5, sch)
    r = api.sampler_run(20000, 4, _target(api, gmm, K, 0.8), 31, mode, drafter)
    assert np.all(r["k"].cpu().numpy() == K)
    _check_law(r["y"].cpu().numpy().astype(np.float64), m, var)


def test_gpu_speculative_and_em_agree_on_the_mixture(api):
    cfg = W.SAMPLER_CONFIG
    d = 16
    gmm = _gmm(8, d, 7)
    K = 100
    tgt = _target(api, gmm, K, cfg["churn"])
    n = 8000
    y_em = api.em_sample(n, tgt, 41).cpu().numpy()
    rng = np.random.Generator(np.random.PCG64(8))
    dirs = rng.standard_normal((4, d))
    for mode in ("sample", "block"):
        r = api.sampler_run(n, 8, tgt, 42, mode)
        y = r["y"].cpu().numpy()
        for u in dirs:
            assert stats.ks_2samp(y_em @ u, y @ u).pvalue > 1e-3
        # mean accepted steps per parallel target call is at least one
        assert r["tau_sum"].cpu().numpy().sum() >= n * K
