"""fp64 oracle of the end-to-end speculative diffusion sampler (test infrastructure only).

Plain numpy, vectorised over chains; every step follows the paper:

* forward SDE dX = f_t X dt + g_t dB with q_1 = N(0, I) (Eq. forward-process); here the
  variance-preserving schedule beta(t) = beta_min + (beta_max - beta_min) t,
  f_t = -beta(t)/2, g_t = sqrt(beta(t)), alpha_bar_t = exp(-int_0^t beta);
* generative drift b_t(y) = -f_{1-t} y + (1 + eps^2)/2 g_{1-t}^2 s_{1-t}(y), churn eps
  (Eq. backward-process);
* Euler-Maruyama target kernel q(y_{k+1} | y_k) = N(m^q_k(y_k), sigma_k^2 I),
  m^q_k(y) = y + delta b_{t_k}(y), sigma_k = sqrt(delta) eps g_{1-t_k}, t_k = k delta,
  delta = 1/K (Eq. target-distribution); the forward time 1 - t_k is floored at t_floor;
* drafter p with the same sigma_k and mean m^p (Eq. draft-distribution):
  Frozen drafter (Eq. frozen-draft-drift): b^p(yhat) = -f yhat + (1+eps^2)/2 g^2 s^q_{1-t_k}(y_k),
  one fresh score per round; Free drafter (Sec. "Self-Speculative Drafter"): the same drift
  with the score reused from the previous round's parallel verification (the score at the
  state that becomes the next round's start index, or at the last draft on a full accept);
  the target is called explicitly only before the first round;
* one round (Alg. abstract-spec-diffusion / full-block-verification): gamma_k = min(gamma,
  K - k); draft gamma_k steps; target means at yhat_{k..k+gamma_k} in parallel; verification
  (oracle.verify); residual or bonus step (only while k + tau <= K); accept the prefix;
  k = min(k + tau, K).

The analytic target is a Gaussian mixture q_data = sum_c w_c N(mu_c, s^2 I), so
q_t = sum_c w_c N(sqrt(abar_t) mu_c, (abar_t s^2 + 1 - abar_t) I) and its score is
s_t(x) = sum_c r_c(x) (sqrt(abar_t) mu_c - x) / v_t with r = softmax(log w_c - |x - sqrt(abar_t)
mu_c|^2 / (2 v_t)).

Random numbers (each side implements the same Philox layout): the initial state Y_0 from
stream 5 with the base seed; round r uses seed_r = round_seed(seed, r) for the draft noise
(stream 4, sub-counter = draft step index) and inside verification; the plain EM chain
draws step k from stream 6 (sub-counter k) with the base seed.
"""
import math

import numpy as np

from . import philox
from . import verify as V


class VPSchedule:
    def __init__(self, K, churn, beta_min=0.1, beta_max=20.0, t_floor=1e-4):
        self.K = int(K)
        self.churn = float(churn)
        self.beta_min = float(beta_min)
        self.beta_max = float(beta_max)
        self.t_floor = float(t_floor)
        self.delta = 1.0 / self.K

    def tfwd(self, k):
        """Forward time 1 - t_k of generative step k (floored)."""
        return np.maximum(1.0 - np.asarray(k, dtype=np.float64) * self.delta, self.t_floor)

    def beta(self, tf):
        return self.beta_min + (self.beta_max - self.beta_min) * tf

    def alpha_bar(self, tf):
        return np.exp(-(self.beta_min * tf + 0.5 * (self.beta_max - self.beta_min) * tf * tf))

    def sigma(self, k):
        """sigma_k = sqrt(delta) * eps * g_{1-t_k}."""
        return math.sqrt(self.delta) * self.churn * np.sqrt(self.beta(self.tfwd(k)))


def gmm_score(x, tf, means, log_w, comp_var, sched):
    """Score of q_tf at x (rows), for the mixture sum_c w_c N(mu_c, comp_var I)."""
    x = np.asarray(x, dtype=np.float64)
    tf = np.broadcast_to(np.asarray(tf, dtype=np.float64), x.shape[:-1])
    ab = sched.alpha_bar(tf)
    v = ab * comp_var + 1.0 - ab
    centers = np.sqrt(ab)[..., None, None] * np.asarray(means, dtype=np.float64)   # [..., C, d]
    d2 = np.sum((x[..., None, :] - centers) ** 2, axis=-1)                         # [..., C]
    logits = np.asarray(log_w, dtype=np.float64) - d2 / (2.0 * v[..., None])
    logits -= logits.max(axis=-1, keepdims=True)
    r = np.exp(logits)
    r /= r.sum(axis=-1, keepdims=True)
    return (np.sum(r[..., None] * centers, axis=-2) - x) / v[..., None]


def target_mean(y, k, gmm, sched):
    """m^q_k(y) = y + delta [beta/2 y + (1 + eps^2)/2 beta s_{1-t_k}(y)] and the score used."""
    y = np.asarray(y, dtype=np.float64)
    tf = sched.tfwd(k)
    b = sched.beta(tf)
    s = gmm_score(y, tf, gmm["means"], gmm["log_weights"], gmm["comp_var"], sched)
    bb = np.broadcast_to(b, y.shape[:-1])[..., None]
    drift = 0.5 * bb * y + 0.5 * (1.0 + sched.churn ** 2) * bb * s
    return y + sched.delta * drift, s


def initial_state(seed, B, d):
    return philox.normals(seed, np.arange(B), d, philox.STREAM_INIT)


def em_sample(B, d, gmm, sched, seed, chains=None):
    """Plain Euler-Maruyama chain (the non-speculative baseline): Y_{k+1} = m^q_k(Y_k) + sigma_k G_k."""
    chains = np.arange(B) if chains is None else np.asarray(chains)
    y = philox.normals(seed, chains, d, philox.STREAM_INIT)
    for k in range(sched.K):
        mq, _ = target_mean(y, np.full(len(chains), k), gmm, sched)
        G = philox.normals(seed, chains, d, philox.STREAM_EM, sub=k)
        y = mq + float(sched.sigma(k)) * G
    return y


def draft(y, s_cache, k, g, L, sched, seed_r, chains):
    """Draft gamma_k = g steps from y with the cached score (Free / Frozen drafter mean).

    Returns x_draft [n, L, d] (yhat_{k+1..k+L}), mu_draft [n, L, d] (m^p_{k..k+L-1}) and
    sigma [n, L]; rows j >= g are zero (never read).
    """
    n, d = y.shape
    x = np.zeros((n, L, d))
    mp = np.zeros((n, L, d))
    sg = np.zeros((n, L))
    cur = y.copy()
    c = 0.5 * (1.0 + sched.churn ** 2)
    for i in range(1, L + 1):
        live = i <= g
        kk = k + i - 1
        b = sched.beta(sched.tfwd(kk))[:, None]
        m = cur + sched.delta * (0.5 * b * cur + c * b * s_cache)
        s_i = sched.sigma(kk)
        G = philox.normals(seed_r, chains, d, philox.STREAM_DRAFT, sub=i - 1)
        nxt = m + s_i[:, None] * G
        mp[live, i - 1] = m[live]
        x[live, i - 1] = nxt[live]
        sg[live, i - 1] = s_i[live]
        cur = np.where(live[:, None], nxt, cur)
    return x, mp, sg


def speculative_sample(B, d, L, mode, gmm, sched, seed, drafter="free", chains=None,
                       max_rounds=None, return_trace=False):
    """Speculative sampling with sample (mode 0) or block (mode 1) verification.

    Returns dict(y = Y_K [n, d], rounds = number of rounds, chain_rounds [n] = rounds in which
    each chain took part, taus = list of tau arrays per round, target_calls = parallel target
    calls (initial score + one per round, + one per round for the Frozen drafter)).
    """
    chains = np.arange(B) if chains is None else np.asarray(chains)
    n = len(chains)
    K = sched.K
    y = philox.normals(seed, chains, d, philox.STREAM_INIT)
    k = np.zeros(n, dtype=np.int64)
    _, s_cache = target_mean(y, k, gmm, sched)          # the only explicit target call
    target_calls = 1
    rounds = 0
    chain_rounds = np.zeros(n, dtype=np.int64)
    taus = []
    trace = []
    while np.any(k < K) and (max_rounds is None or rounds < max_rounds):
        seed_r = philox.round_seed(seed, rounds)
        active = k < K
        g = np.where(active, np.minimum(L, K - k), 0)
        if drafter == "frozen":
            _, s_fresh = target_mean(y, k, gmm, sched)
            s_cache = np.where(active[:, None], s_fresh, s_cache)
            target_calls += 1
        x, mp, sg = draft(y, s_cache, k, g, L, sched, seed_r, chains)
        # parallel target call on yhat_k .. yhat_{k+g}
        states = np.concatenate([y[:, None], x], axis=1)            # [n, L+1, d]
        kk = k[:, None] + np.arange(L + 1)[None, :]
        mq_all, sc_all = target_mean(states, kk, gmm, sched)
        target_calls += 1
        mq = mq_all[:, :L]
        rows = np.arange(n)
        mq_bonus = mq_all[rows, g]
        s_bonus = sched.sigma(k + g)
        res = V.verify(x, mq, mp, np.where(sg > 0, sg, 1.0), seed_r, mode, Leff=g,
                       mu_target_bonus=mq_bonus, sigma_bonus=s_bonus,
                       chain_ids=chains)
        tau = res["tau"]
        # chains whose window reaches the end take no bonus step: they stop at yhat_{k+g}
        end = active & (tau == g + 1) & (k + g >= K)
        y_new = np.where(end[:, None], x[rows, np.maximum(g - 1, 0)], res["y"])
        y = np.where(active[:, None], y_new, y)
        idx = np.minimum(tau, g)
        s_cache = np.where(active[:, None], sc_all[rows, idx], s_cache)
        k = np.where(active, np.minimum(k + tau, K), k)
        chain_rounds += active
        taus.append(np.where(active, tau, 0))
        if return_trace:
            trace.append(dict(k=k.copy(), y=y.copy(), tau=tau.copy(), g=g.copy(), res=res,
                              x_draft=x, mu_draft=mp, mu_target=mq, sigma=sg))
        rounds += 1
    out = dict(y=y, rounds=rounds, chain_rounds=chain_rounds, taus=taus,
               target_calls=target_calls, k=k)
    if return_trace:
        out["trace"] = trace
    return out


def linear_gaussian_moments(mu, comp_var, sched):
    """Mean vector and per-coordinate variance of Y_K of the EM chain for a one-component
    target (the chain is linear: Y_{k+1} = a_k Y_k + c_k + sigma_k G_k, Y_0 ~ N(0, I))."""
    mu = np.asarray(mu, dtype=np.float64)
    m = np.zeros_like(mu)
    var = 1.0
    cst = 0.5 * (1.0 + sched.churn ** 2)
    for k in range(sched.K):
        tf = float(sched.tfwd(k))
        b = float(sched.beta(tf))
        ab = float(sched.alpha_bar(tf))
        v = ab * comp_var + 1.0 - ab
        a = 1.0 + sched.delta * (0.5 * b - cst * b / v)
        c = sched.delta * cst * b * math.sqrt(ab) * mu / v
        s = float(sched.sigma(k))
        m = a * m + c
        var = a * a * var + s * s
    return m, var
