"""Shared helpers of the GPU parity tests: move seeded inputs to the device, run the
C-ABI path and the oracle on the same inputs, and compare with the stated tolerances.

Tolerances (from the verification step's accuracy targets):
  * log ratios and |Delta|: |gpu - oracle| <= 1e-5 * max(1, |oracle|);
  * accepted lengths: bit-exact, except for a chain whose oracle run has a coin
    within the tie band of its threshold: |log eta_j - log thr_j| < 1e-4 plus the
    propagated log-ratio tolerance (thr = min{1, e^ell} in sample mode, h_j in block
    mode, where log alpha_j accumulates the tolerance of ell_1..ell_j);
  * output states (chains with equal tau): 1e-5 absolute for fp32 inputs, 2e-2 for bf16
    (widened to half a bf16 ulp where |y| > 5.12; y_tolerance).
"""
import numpy as np
import torch

from oracle import philox as OP
from oracle import verify as OV

TOL_Y = {"f32": 1e-5, "bf16": 2e-2}


def y_tolerance(y_ref, dtype):
    """Output-state tolerance: 1e-5 absolute for fp32; 2e-2 absolute for bf16, widened
    to the output's own rounding, half a bf16 ulp (at most 2^-8 |y|), where |y| > 5.12:
    a bf16 state of magnitude 8 or more is 0.0625 from its neighbours, so no
    implementation that stores y in bf16 can be within 2e-2 of every value there."""
    if dtype == "bf16":
        return np.maximum(TOL_Y["bf16"], 2.0 ** -8 * np.abs(y_ref))
    return TOL_Y[dtype]


def to_dev(inp, name):
    if inp["dtype"] == "bf16":
        bits = np.ascontiguousarray(inp[name + "_bits"]).view(np.int16)
        return torch.from_numpy(bits).cuda().view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(inp[name])).cuda()


def run_gpu(api, inp, seed, mode, sigma=None, **kw):
    x = to_dev(inp, "x_draft")
    mq = to_dev(inp, "mu_target")
    mp = to_dev(inp, "mu_draft")
    sg = torch.from_numpy(np.ascontiguousarray(inp["sigma"] if sigma is None else sigma)).cuda()
    dev_kw = {}
    for k, v in kw.items():
        if isinstance(v, np.ndarray):
            v = torch.from_numpy(np.ascontiguousarray(v)).cuda()
        dev_kw[k] = v
    if "mu_target_bonus" in dev_kw and inp["dtype"] == "bf16":
        dev_kw["mu_target_bonus"] = dev_kw["mu_target_bonus"].to(torch.bfloat16)
    r = api.verify(x, mq, mp, sg, seed, mode, with_aux=True, **dev_kw)
    torch.cuda.synchronize()
    out = {k: (v.float().cpu().numpy() if v.dtype == torch.bfloat16 else v.cpu().numpy())
           for k, v in r.items()}
    return out


def near_tie(o, mode, omega=1.0, band=1e-4, rtol=1e-5):
    """Per chain: does the oracle run have a coin inside the tie band of its threshold?"""
    ell = o["ell"] / (omega * omega)
    leta = np.log(o["eta"])
    slack = rtol * np.maximum(1.0, np.abs(o["ell"])) / (omega * omega)
    n, L = ell.shape
    if mode == OV.MODE_SAMPLE:
        thr = np.minimum(0.0, ell)
        tie = np.abs(leta - thr) < band + slack
    else:
        with np.errstate(divide="ignore"):
            lh = np.log(o["h"][:, 1:])
        cum = np.cumsum(slack, axis=1)
        tie = np.abs(leta - lh) < band + cum
        # h_j is discontinuous at alpha_j = 1 when |Delta_{j+1}| = 0 (h = 1 at alpha = 1,
        # h = 0 for any alpha < 1): a log alpha_j within rounding of 0 there is a tie
        la = np.zeros((n, L))
        run = np.zeros(n)
        for j in range(L):
            run = np.minimum(0.0, run + ell[:, j])
            la[:, j] = run
        dnext = np.concatenate([o["dnorm"][:, 1:], np.ones((n, 1))], axis=1) \
            if "dnorm" in o else np.ones((n, L))
        tie |= (dnext == 0.0) & (np.abs(la) < 1e-5 * (1 + np.arange(L)))
    return tie.any(axis=1)


def ell_error_bound(inp, chains=None, gamma=128 * 2.0 ** -24):
    """Per (chain, step) bound on the fp32 error of the log ratio.

    ell = -(S1 + S2/2)/sigma^2 with S1 = sum (x - m^p)(m^p - m^q) and S2 = sum (m^p - m^q)^2
    summed in fp32: any summation order of n terms errs by at most about n_levels ulps of
    the sum of the terms' magnitudes, T = (sum |a_i delta_i| + sum delta_i^2 / 2)/sigma^2,
    not of |ell| itself, which can be far smaller than T when S1 and S2/2 cancel (a
    relative tolerance on ell is ill-posed there).  128 ulps covers the kernels'
    orders (a thread's sequential sweep, a warp and CTA tree, a sequential sum over
    the row's tiles) for rows up to the largest workload's 196608 elements."""
    ch = np.arange(np.shape(inp["x_draft"])[0]) if chains is None else np.asarray(chains)
    x = inp["x_draft"][ch].astype(np.float64)
    mq = inp["mu_target"][ch].astype(np.float64)
    mp = inp["mu_draft"][ch].astype(np.float64)
    dl = mp - mq
    T = (np.sum(np.abs((x - mp) * dl), axis=-1) + 0.5 * np.sum(dl * dl, axis=-1))
    B, L = np.shape(inp["x_draft"])[:2]
    T /= np.broadcast_to(np.asarray(inp["sigma"], np.float64), (B, L))[ch] ** 2
    return gamma * T


def compare(g, o, mode, dtype, omega=1.0, max_tie_frac=0.05):
    """Assert parity of a GPU result dict with an oracle result dict (same chains).

    Log ratios: within 1e-5 relative (1e-5 absolute where |ell| < 1), and, where the
    oracle dict carries it, within the fp32 error bound of the reduction
    (ell_error_bound), which holds the relative tolerance wherever S1 and S2/2 do not
    cancel."""
    ell_g, ell_o = g["log_ratio"], o["ell"]
    err = np.abs(ell_g - ell_o)
    assert np.all(err <= 1e-5 * np.maximum(1.0, np.abs(ell_o))), \
        "log ratio max err %g" % np.max(err / np.maximum(1.0, np.abs(ell_o)))
    if "ell_bound" in o:
        bound = o["ell_bound"] + 4 * 2.0 ** -24 * np.abs(ell_o)
        assert np.all(err <= bound), "log ratio error above its fp32 bound: %g" % np.max(err / bound)
    dn_g, dn_o = g["delta_norm"], o["dnorm"]
    assert np.all(np.abs(dn_g - dn_o) <= 1e-5 * np.maximum(1.0, dn_o)), "delta norm"
    acc_g, acc_o = g["accepted_len"], o["accepted_len"]
    diff = acc_g != acc_o
    if diff.any():
        ties = near_tie(o, mode, omega)
        assert np.all(ties[diff]), "accepted length differs outside the tie band: chains %s" % \
            np.nonzero(diff & ~ties)[0][:10]
        assert diff.mean() <= max_tie_frac
    same = ~diff
    yg, yo = g["y"][same], o["y"][same]
    act = np.isfinite(yo).all(axis=1)          # inactive chains emit nothing
    err = np.abs(yg[act] - yo[act])
    tol = y_tolerance(yo[act], dtype)
    assert err.size == 0 or np.all(err <= tol), "y max err %g (tol %g)" % (
        err.max(), tol if np.isscalar(tol) else tol.flat[np.argmax(err)])
    assert np.array_equal(g["status"][same][act] & 3, o["status"][same][act] & 3)
    return int(diff.sum())


def oracle_for(inp, seed, mode, chains=None, **kw):
    o = OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], seed,
                  mode, chains=chains, **kw)
    Leff = kw.get("Leff")
    bound = ell_error_bound(inp, chains)
    if Leff is not None:
        g = np.asarray(Leff)[o["chains"]]
        bound = np.where(np.arange(bound.shape[1])[None, :] < g[:, None], bound, 0.0)
    o["ell_bound"] = bound
    return o


def philox_words(ctr, seed):
    k0, k1 = OP.key_of(seed)
    w = OP.philox4x32_10(ctr[:, 0], ctr[:, 1], ctr[:, 2], ctr[:, 3], k0, k1)
    return np.stack(w, axis=1).astype(np.uint32)
