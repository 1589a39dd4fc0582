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


@pytest.mark.parametrize("d", [1024, 37])
def test_gmm_target_matches_oracle(api, d):
    gmm = _gmm(8, d, 1)
    K = 1000
    sch = OS.VPSchedule(K, 0.5)
    rng = np.random.Generator(np.random.PCG64(2))
    n = 96
    k = rng.integers(0, K + 1, n).astype(np.int32)
    tf = sch.tfwd(k)
    ab = sch.alpha_bar(tf)
    # states near the noised mixture at their own step, plus generic points
    comp = rng.integers(0, 8, n)
    z = (np.sqrt(ab)[:, None] * gmm["means"][comp]
         + np.sqrt(ab * gmm["comp_var"] + 1 - ab)[:, None] * rng.standard_normal((n, d)))
    z[::7] = 3.0 * rng.standard_normal((len(z[::7]), d))
    z = z.astype(np.float32)
    mq, sc = api.gmm_target(torch.from_numpy(z).cuda(), torch.from_numpy(k).cuda(),
                            _target(api, gmm, K, 0.5))
    mq, sc = mq.cpu().numpy(), sc.cpu().numpy()
    mq_o, sc_o = OS.target_mean(z, k, gmm, sch)
    assert np.max(np.abs(mq - mq_o) / np.maximum(1.0, np.abs(mq_o))) < 2e-5
    scale = np.maximum(1.0, np.abs(sc_o).max(axis=1, keepdims=True))
    assert np.max(np.abs(sc - sc_o) / scale) < 2e-3


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
    assert np.max(np.abs(x - xo)[live]) < 2e-5
    assert np.max(np.abs(mp - mpo)[live]) < 2e-5
    assert np.max(np.abs(sg - sgo)[live] / sgo[live]) < 1e-5


def test_em_chain_matches_oracle(api):
    d, Bn, K = 64, 32, 12
    gmm = _gmm(8, d, 5)
    sch = OS.VPSchedule(K, 0.5)
    y = api.em_sample(Bn, _target(api, gmm, K, 0.5), 9).cpu().numpy()
    yo = OS.em_sample(Bn, d, gmm, sch, 9)
    assert np.max(np.abs(y - yo) / np.maximum(1.0, np.abs(yo))) < 1e-4


def _first_rounds(api, mode, drafter, d, C, Bn=192, L=4, K=40):
    gmm = _gmm(C, d, 6)
    sch = OS.VPSchedule(K, 0.5)
    tgt = _target(api, gmm, K, 0.5)
    o = OS.speculative_sample(Bn, d, L, mode, gmm, sch, seed=123, drafter=drafter, max_rounds=3,
                              return_trace=True)
    clean = np.ones(Bn, dtype=bool)
    for R in (1, 2, 3):
        r = api.sampler_run(Bn, L, tgt, 123, "block" if mode else "sample", drafter, max_rounds=R)
        assert r["rounds"] == R
        tr = o["trace"][R - 1]
        res = tr["res"]
        clean &= ~near_tie(res, mode)
        k = r["k"].cpu().numpy()
        y = r["y"].cpu().numpy()
        assert clean.mean() > 0.9
        np.testing.assert_array_equal(k[clean], tr["k"][clean])
        err = np.abs(y[clean] - tr["y"][clean]) / np.maximum(1.0, np.abs(tr["y"][clean]))
        assert err.max() < 1e-4, err.max()


@pytest.mark.parametrize("mode", [OV.MODE_SAMPLE, OV.MODE_BLOCK])
@pytest.mark.parametrize("drafter", ["free", "frozen"])
def test_first_rounds_match_oracle(api, mode, drafter):
    """Rounds 1..3 element by element: k, and the states of chains whose coins all lie
    outside the tie band in every round so far."""
    _first_rounds(api, mode, drafter, 64, 8)


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
