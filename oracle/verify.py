"""fp64 oracle of the verification step of speculative diffusion sampling.

Test infrastructure only (see ``oracle/__init__``).  Plain numpy/scipy, float64,
vectorised over independent chains only; every step is the paper's, in the
paper's order and notation:

  Delta_j = (m^p_{k+j-1} - m^q_{k+j-1}) / sigma_{k+j-1},
  Z_j     = (yhat_{k+j} - m^p_{k+j-1}) / sigma_{k+j-1}            (Alg. token-/block-verification)
  log N(Z+Delta)/N(Z) = -Z^T Delta - |Delta|^2 / 2                 (App. A.2, density ratios)
  sample verification: alpha_j = min{1, ratio_j}, c_j = [eta < alpha_j],
      tau = first j with c_j = 0, else gamma+1; alpha_res = 1       (Alg. token-verification)
  block verification: log alpha_j = min{0, log alpha_{j-1} + log ratio_j},
      h_j = v_j / (v_j + 1 - alpha_j) for j < gamma, h_gamma = alpha_gamma,
      v_j = alpha_j Phi(log alpha_j/|Delta_{j+1}| + |Delta_{j+1}|/2)
            - Phi(log alpha_j/|Delta_{j+1}| - |Delta_{j+1}|/2),
      c_j = [eta < h_j], tau = 1 + max{j in 0..gamma : c_j = 1} (c_0 = 1),
      alpha_res = alpha_{tau-1}                                       (Alg. block-verification)
  Psi_alpha(u) = (alpha Phi(u) - Phi(u - |Delta|)) / v  for u < a+, else 1,
      a+ = log alpha/|Delta| + |Delta|/2                              (Prop. decomposition, Eq. u-cdf)
  U = Psi_alpha^{-1}(w) by bracketing + bisection                     (Alg. u-sample)
  Y = m^q + sigma (U e + G - e (e^T G)), e = Delta/|Delta|            (Alg. decomposition-res)
  Y = m^q + sigma (I - 2 e e^T) Z                                     (Alg. reflect-res)
  temperature omega: the density ratio uses N(.; 0, omega^2 I), i.e.
      log ratio / omega^2; h_j and the residual take the tempered alpha (App. Temperature,
      Alg. token-/block-verification-temperature)

Differences of CDFs are evaluated with log-CDF primitives and a stable
log-sub-exp, as App. A.2 recommends.  Phi and log Phi are scipy's ndtr /
log_ndtr (library primitives).

Readings where the paper is silent (identical on the CUDA side):
  * one coin per (chain, step) from Philox stream 0, drawn for every step;
  * the bisection stops when the bracket is narrower than ``xtol * max(1, |mid|)``
    (the paper's |Psi(mid) - w| <= tol with tol -> 0); no 3/4-iteration caps;
  * degenerate h_j: alpha_j = 1 -> 1; alpha_j = 0 or |Delta_{j+1}| = 0 (alpha_j < 1) -> 0;
  * |Delta_tau| = 0 at the residual (probability zero): Y = m^q + sigma G, status bit 1;
  * full accept without a bonus mean returns the last draft row; with one,
    Y = m^q_bonus + sigma_bonus G_bonus (Alg. abstract-spec-diffusion bonus step).
"""
import math

import numpy as np
from scipy.special import log_ndtr

from . import philox

MODE_SAMPLE = 0
MODE_BLOCK = 1
RESIDUAL_DECOMPOSITION = 0
RESIDUAL_REFLECTION = 1

STATUS_ZERO_DELTA = 1
STATUS_NONFINITE = 2

LN2 = math.log(2.0)


def log1mexp(x):
    """log(1 - e^x) for x <= 0 (stable log-sub-exp building block)."""
    x = np.asarray(x, dtype=np.float64)
    with np.errstate(divide="ignore", invalid="ignore"):
        return np.where(x > -LN2, np.log(-np.expm1(x)), np.log1p(-np.exp(x)))


# --------------------------------------------------------------------------
# Log density ratios (App. A.2) - vectorised over any leading dimensions.
# --------------------------------------------------------------------------
def delta_and_z(x, mu_target, mu_draft, sigma):
    """Delta = (m^p - m^q)/sigma and Z = (yhat - m^p)/sigma for rows [..., d]; sigma [...]."""
    x = np.asarray(x, dtype=np.float64)
    mq = np.asarray(mu_target, dtype=np.float64)
    mp = np.asarray(mu_draft, dtype=np.float64)
    s = np.asarray(sigma, dtype=np.float64)[..., None]
    return (mp - mq) / s, (x - mp) / s


def log_ratios(x, mu_target, mu_draft, sigma):
    """ell = log N(Z+Delta; 0, I)/N(Z; 0, I) = -Z^T Delta - |Delta|^2/2 and D = |Delta|."""
    Delta, Z = delta_and_z(x, mu_target, mu_draft, sigma)
    DD = np.sum(Delta * Delta, axis=-1)
    ell = -np.sum(Z * Delta, axis=-1) - 0.5 * DD
    return ell, np.sqrt(DD)


# --------------------------------------------------------------------------
# Verification rules, vectorised over chains (the loop over steps j is explicit).
# ell, dnorm, eta: [B, L]; Leff: [B] (window length gamma_k <= L).
# --------------------------------------------------------------------------
def sample_verification(ell, eta, Leff, omega=1.0):
    """Alg. token-verification (and its temperature variant): returns tau [B] (1-based)."""
    ell = np.asarray(ell, dtype=np.float64) / (omega * omega)
    B, L = ell.shape
    Leff = np.asarray(Leff)
    tau = Leff.astype(np.int64) + 1                 # gamma+1 unless a coin fails
    undecided = np.ones(B, dtype=bool)
    for j in range(1, L + 1):
        live = undecided & (j <= Leff)
        alpha_j = np.exp(np.minimum(0.0, ell[:, j - 1]))      # min{1, ratio_j}
        c_j = eta[:, j - 1] < alpha_j
        fail = live & ~c_j
        tau[fail] = j
        undecided &= ~fail
    return tau


def log_residual_mass(log_alpha, D):
    """log v, v = alpha Phi(log alpha/D + D/2) - Phi(log alpha/D - D/2) = int max{0, alpha q - p}.

    Requires D > 0 and log alpha finite.  Written as
    log v = log alpha + log Phi(a+) + log(1 - exp(log Phi(a-) - log alpha - log Phi(a+))).
    """
    la = np.asarray(log_alpha, dtype=np.float64)
    D = np.asarray(D, dtype=np.float64)
    a_plus = la / D + 0.5 * D
    a_minus = la / D - 0.5 * D
    lp = log_ndtr(a_plus)
    lm = log_ndtr(a_minus)
    return la + lp + log1mexp(np.minimum(lm - la - lp, 0.0))


def block_h(log_alpha_j, D_next):
    """h_j = v_j / (v_j + 1 - alpha_j), v_j from alpha_j and |Delta_{j+1}| (arrays).

    Degenerate limits: alpha_j = 1 -> 1 (1 - alpha_j = 0); alpha_j = 0 or
    |Delta_{j+1}| = 0 with alpha_j < 1 -> 0 (v_j = 0 < 1 - alpha_j).
    """
    la = np.asarray(log_alpha_j, dtype=np.float64)
    Dn = np.asarray(D_next, dtype=np.float64)
    regular = (la < 0.0) & np.isfinite(la) & (Dn > 0.0)
    la_r = np.where(regular, la, -1.0)
    D_r = np.where(regular, Dn, 1.0)
    lv = log_residual_mass(la_r, D_r)
    l1ma = log1mexp(la_r)                             # log(1 - alpha_j)
    h = np.exp(lv - np.logaddexp(lv, l1ma))
    return np.where(regular, h, np.where(la == 0.0, 1.0, 0.0))


def block_verification(ell, dnorm, eta, Leff, omega=1.0):
    """Alg. block-verification (and its temperature variant).

    Returns tau [B] (1-based), log alpha_res [B] = log alpha_{tau-1},
    log_alpha [B, L+1] (column 0 is alpha_0 = 1) and h [B, L+1] (column 0 is c_0's 1).
    """
    ell = np.asarray(ell, dtype=np.float64) / (omega * omega)
    dnorm = np.asarray(dnorm, dtype=np.float64)
    B, L = ell.shape
    Leff = np.asarray(Leff)
    log_alpha = np.zeros((B, L + 1))
    for j in range(1, L + 1):
        log_alpha[:, j] = np.minimum(0.0, log_alpha[:, j - 1] + ell[:, j - 1])
    h = np.zeros((B, L + 1))
    h[:, 0] = 1.0
    last_success = np.zeros(B, dtype=np.int64)       # c_0 = 1
    for j in range(1, L + 1):
        live = j <= Leff
        D_next = dnorm[:, j] if j < L else np.zeros(B)
        h_mid = block_h(log_alpha[:, j], D_next)      # j != gamma_k
        h_end = np.exp(log_alpha[:, j])               # j == gamma_k: h = alpha_gamma
        h[:, j] = np.where(live, np.where(j == Leff, h_end, h_mid), 0.0)
        c_j = live & (eta[:, j - 1] < h[:, j])
        last_success[c_j] = j
    tau = 1 + last_success
    la_res = log_alpha[np.arange(B), tau - 1]
    return tau, la_res, log_alpha, h


# --------------------------------------------------------------------------
# Residual: Psi_alpha, USampleViaBisection, decomposition and reflection.
# --------------------------------------------------------------------------
def psi_cdf(u, D, log_alpha):
    """Psi_alpha(u) of Eq. u-cdf (arrays), in log space."""
    u = np.asarray(u, dtype=np.float64)
    D = np.asarray(D, dtype=np.float64)
    la = np.asarray(log_alpha, dtype=np.float64)
    a_plus = la / D + 0.5 * D
    below = u < a_plus
    ub = np.where(below, u, a_plus - 1.0)
    lu = log_ndtr(ub)
    lum = log_ndtr(ub - D)
    lnum = la + lu + log1mexp(np.minimum(lum - la - lu, 0.0))
    lden = log_residual_mass(la, D)
    return np.where(below, np.minimum(1.0, np.exp(lnum - lden)), 1.0)


def usample_bisection(D, log_alpha, w, tol=0.0, xtol=1e-12):
    """Alg. u-sample, for arrays of independent (|Delta|, log alpha, w).

    Bounds (a+ - 1, a+); while Psi(lower) > w the lower bound becomes
    upper - 2 (upper - lower); then bisection on the sign of Psi(mid) - w until
    |Psi(mid) - w| <= tol or the bracket is narrower than xtol * max(1, |mid|)
    (the paper leaves tol unspecified; a relative width keeps the loop finite
    where the fp64 spacing of |mid| exceeds xtol).
    """
    D = np.atleast_1d(np.asarray(D, dtype=np.float64))
    la = np.atleast_1d(np.asarray(log_alpha, dtype=np.float64))
    w = np.atleast_1d(np.asarray(w, dtype=np.float64))
    a_plus = la / D + 0.5 * D
    lo, hi = a_plus - 1.0, a_plus.copy()
    grow = psi_cdf(lo, D, la) > w
    while np.any(grow):
        lo = np.where(grow, hi - 2.0 * (hi - lo), lo)
        grow = psi_cdf(lo, D, la) > w
    mid = 0.5 * (lo + hi)
    active = np.ones(D.shape, dtype=bool)
    while True:
        p = psi_cdf(mid, D, la)
        active &= ~((np.abs(p - w) <= tol) | ((hi - lo) <= xtol * np.maximum(1.0, np.abs(mid))))
        if not np.any(active):
            break
        lo = np.where(active & (p < w), mid, lo)
        hi = np.where(active & (p >= w), mid, hi)
        mid = np.where(active, 0.5 * (lo + hi), mid)
    return mid


def decomposition_residual(Delta, mq, sigma, U, G):
    """Alg. decomposition-res on rows [n, d]: Y = m^q + sigma (U e + Z_perp), Z_perp = G - e (e^T G)."""
    e = Delta / np.sqrt(np.sum(Delta * Delta, axis=-1, keepdims=True))
    Z_perp = G - e * np.sum(e * G, axis=-1, keepdims=True)
    return mq + sigma[:, None] * (U[:, None] * e + Z_perp)


def reflection_residual(Delta, Z, mq, sigma):
    """Alg. reflect-res on rows [n, d]: Y = m^q + sigma (I - 2 e e^T) Z."""
    e = Delta / np.sqrt(np.sum(Delta * Delta, axis=-1, keepdims=True))
    return mq + sigma[:, None] * (Z - 2.0 * e * np.sum(e * Z, axis=-1, keepdims=True))


# --------------------------------------------------------------------------
# The whole verification step for B chains (the semantics of the C-ABI sdv_verify_ex).
# --------------------------------------------------------------------------
def verify(x_draft, mu_target, mu_draft, sigma, seed, mode, Leff=None,
           mu_target_bonus=None, sigma_bonus=None, residual=RESIDUAL_DECOMPOSITION,
           omega=1.0, chains=None, xtol=1e-12, chain_ids=None):
    """Run the verification step on chains ``chains`` (default: all) of a [B, L, d] window.

    x_draft: yhat_{k+1..k+L}; mu_target: m^q_{k..k+L-1}; mu_draft: m^p_{k..k+L-1};
    sigma: [B, L] (sigma_{k..k+L-1}).  Arrays may be any float dtype (widened to fp64).
    Leff: [B] window lengths gamma_k (default L; 0 marks an inactive chain).
    chain_ids: the chain indices that key the random numbers of the selected rows
    (default: ``chains`` itself); a caller that holds a subset of a larger batch in
    compact arrays passes the subset's indices in the full batch here.
    Returns a dict of per-chain results for the selected chains, in the order given.
    """
    x_draft = np.asarray(x_draft)
    B, L, d = x_draft.shape
    sigma = np.broadcast_to(np.asarray(sigma, dtype=np.float64), (B, L))
    Leff = np.full(B, L, dtype=np.int64) if Leff is None else np.asarray(Leff, dtype=np.int64)
    chains = np.arange(B) if chains is None else np.asarray(chains, dtype=np.int64)
    n = len(chains)
    g = Leff[chains]
    ids = chains if chain_ids is None else np.asarray(chain_ids, dtype=np.int64)
    assert len(ids) == n

    xs = np.asarray(x_draft[chains], dtype=np.float64)
    mqs = np.asarray(np.asarray(mu_target)[chains], dtype=np.float64)
    mps = np.asarray(np.asarray(mu_draft)[chains], dtype=np.float64)
    sg = sigma[chains]
    ell, dnorm = log_ratios(xs, mqs, mps, sg)
    in_window = np.arange(L)[None, :] < g[:, None]
    ell = np.where(in_window, ell, 0.0)
    dnorm = np.where(in_window, dnorm, 0.0)
    status = np.zeros(n, dtype=np.int64)
    bad = ~(np.isfinite(ell) & np.isfinite(dnorm)).all(axis=1)
    status[bad] |= STATUS_NONFINITE
    eta = philox.coins(seed, ids, L)

    if mode == MODE_SAMPLE:
        tau = sample_verification(ell, eta, g, omega)
        la_res = np.zeros(n)
        h = None
    else:
        tau, la_res, _, h = block_verification(ell, dnorm, eta, g, omega)

    y = np.full((n, d), np.nan)
    U = np.full(n, np.nan)
    rows = np.arange(n)
    resid = (g > 0) & (tau <= g)
    r = np.where(resid, tau - 1, 0)
    Delta, Z = delta_and_z(xs[rows, r], mqs[rows, r], mps[rows, r], sg[rows, r])
    mq_r = mqs[rows, r]
    s_r = sg[rows, r]
    Dn = np.sqrt(np.sum(Delta * Delta, axis=-1))
    zero = resid & (Dn == 0.0)
    status[zero] |= STATUS_ZERO_DELTA
    G = philox.normals(seed, ids, d, philox.STREAM_RESID)
    y[zero] = mq_r[zero] + s_r[zero, None] * G[zero]
    dec = resid & ~zero
    if residual == RESIDUAL_REFLECTION:
        y[dec] = reflection_residual(Delta[dec], Z[dec], mq_r[dec], s_r[dec])
    elif np.any(dec):
        w = philox.usample_uniform(seed, ids[dec])
        U[dec] = usample_bisection(Dn[dec], la_res[dec], w, xtol=xtol)
        y[dec] = decomposition_residual(Delta[dec], mq_r[dec], s_r[dec], U[dec], G[dec])
    full = (g > 0) & (tau == g + 1)
    if mu_target_bonus is not None:
        Gb = philox.normals(seed, ids, d, philox.STREAM_BONUS)
        mqb = np.asarray(np.asarray(mu_target_bonus)[chains], dtype=np.float64)
        sb = np.asarray(sigma_bonus, dtype=np.float64)[chains]
        y[full] = mqb[full] + sb[full, None] * Gb[full]
    else:
        last = np.maximum(g - 1, 0)
        y[full] = xs[rows, last][full]
    return dict(chains=chains, tau=tau, accepted_len=np.where(g > 0, tau - 1, 0), ell=ell,
                dnorm=dnorm, eta=eta, h=h, log_alpha_res=la_res, U=U, y=y, status=status)
