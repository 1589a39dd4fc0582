"""Seeded synthetic inputs for the verification step and the sampler workloads.

This module holds input construction only (numpy PCG64 draws, schedules, bf16
rounding); it contains none of the method's arithmetic and is the one module
both the CUDA path's tests/bench and the CPU oracle consume.

The paper's experiments run trained U-Nets on image datasets that are not
available here; these draws stand in for them with the shapes of its pixel and
latent workloads:

* ``tiny``    B=4,   L=4,  d=16,      fp32; x, m^p ~ N(0,1) independent;
              m^q = m^p + delta u, delta/sigma ~ U(0,2); sigma linear 0.5 -> 0.05.
* ``pixel``   B=256, L=8,  d=3*32*32, fp32; |Delta| ~ U(0,3); cosine sigma schedule.
* ``latent``  B=64,  L=16, d=4*64*64, bf16; |Delta| ~ Gamma(shape 2, scale 0.5); cosine.
* ``highres`` B=16,  L=32, d=3*256*256, fp32; |Delta| ~ U(0,4); sigma linear 1.0 -> 0.01.

For pixel/latent/highres: m^p ~ N(0, I); u a uniform random unit vector per
(chain, step); m^q = m^p - sigma_j |Delta| u (so Delta = |Delta| u); the draft
state is drawn from the draft kernel, x = m^p + sigma_j z, z ~ N(0, I).
bf16 inputs are rounded (nearest-even) after generation; the oracle reads the
rounded values.
"""
import math

import numpy as np

VERIFY_CONFIGS = {
    "tiny": dict(B=4, L=4, d=16, dtype="f32", seed=1),
    "pixel": dict(B=256, L=8, d=3 * 32 * 32, dtype="f32", seed=2),
    "latent": dict(B=64, L=16, d=4 * 64 * 64, dtype="bf16", seed=3),
    "highres": dict(B=16, L=32, d=3 * 256 * 256, dtype="f32", seed=4),
}

# End-to-end sampler workload: 8-component isotropic GMM target in d = 1024,
# component means ~ N(0, 4 I), weights ~ Dirichlet(1), component variance 1,
# 1000-step variance-preserving Euler-Maruyama schedule, B = 1024 chains.
SAMPLER_CONFIG = dict(B=1024, d=1024, n_components=8, K=1000, churn=0.5,
                      beta_min=0.1, beta_max=20.0, t_floor=1e-4, comp_var=1.0, seed=5)


def sigma_schedule(kind, L):
    """Per-step sigma over a window of L steps."""
    j = np.arange(L, dtype=np.float64)
    den = max(L - 1, 1)
    if kind == "tiny":
        s = 0.5 + (0.05 - 0.5) * j / den
    elif kind in ("pixel", "latent"):
        s = 0.05 + 0.95 * 0.5 * (1.0 + np.cos(np.pi * j / den))
    elif kind == "highres":
        s = 1.0 + (0.01 - 1.0) * j / den
    else:
        raise ValueError(kind)
    return s.astype(np.float32)


def round_to_bf16(a):
    """Round float32 values to bfloat16 (nearest, ties to even); returns (uint16 bits, float32 values)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)).astype(np.uint16)
    vals = (r.astype(np.uint32) << np.uint32(16)).view(np.float32)
    return r, vals


def _delta_norms(kind, rng, shape):
    if kind == "pixel":
        return rng.uniform(0.0, 3.0, size=shape)
    if kind == "latent":
        return rng.gamma(2.0, 0.5, size=shape)
    if kind == "highres":
        return rng.uniform(0.0, 4.0, size=shape)
    raise ValueError(kind)


def make_verify_inputs(kind, B=None, L=None, d=None, seed=None, per_chain_sigma=False):
    """Inputs of one verification call for workload ``kind`` (sizes overridable).

    Returns a dict with float32 arrays x_draft, mu_target, mu_draft [B, L, d]
    (for bf16 workloads these hold the bf16-rounded values, and *_bits hold the
    uint16 encodings), sigma [B, L] float32, and the metadata.
    """
    cfg = dict(VERIFY_CONFIGS[kind])
    B = cfg["B"] if B is None else B
    L = cfg["L"] if L is None else L
    d = cfg["d"] if d is None else d
    seed = cfg["seed"] if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    sig_row = sigma_schedule(kind, L)
    sigma = np.broadcast_to(sig_row, (B, L)).copy()
    if per_chain_sigma:
        sigma = (sigma * rng.uniform(0.5, 1.5, size=(B, 1))).astype(np.float32)
    x = np.empty((B, L, d), np.float32)
    mq = np.empty((B, L, d), np.float32)
    mp = np.empty((B, L, d), np.float32)
    for b in range(B):
        s = sigma[b].astype(np.float64)[:, None]
        u = rng.standard_normal((L, d))
        u /= np.linalg.norm(u, axis=1, keepdims=True)
        if kind == "tiny":
            x[b] = rng.standard_normal((L, d))
            mp[b] = rng.standard_normal((L, d))
            delta = s * rng.uniform(0.0, 2.0, size=(L, 1))
            mq[b] = mp[b].astype(np.float64) + delta * u
        else:
            m = rng.standard_normal((L, d))
            Dn = _delta_norms(kind, rng, (L, 1))
            mp[b] = m
            mq[b] = m - s * Dn * u
            x[b] = m + s * rng.standard_normal((L, d))
    out = dict(kind=kind, B=B, L=L, d=d, dtype=cfg["dtype"], sigma=sigma)
    if cfg["dtype"] == "bf16":
        for name, arr in (("x_draft", x), ("mu_target", mq), ("mu_draft", mp)):
            bits, vals = round_to_bf16(arr)
            out[name] = vals.reshape(B, L, d)
            out[name + "_bits"] = bits.reshape(B, L, d)
    else:
        out.update(x_draft=x, mu_target=mq, mu_draft=mp)
    return out


def make_gmm(d=None, n_components=None, seed=None):
    """Analytic Gaussian-mixture target: means [C, d] ~ N(0, 4 I), log-weights [C] of Dirichlet(1)."""
    cfg = SAMPLER_CONFIG
    d = cfg["d"] if d is None else d
    C = cfg["n_components"] if n_components is None else n_components
    seed = cfg["seed"] if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    means = (2.0 * rng.standard_normal((C, d))).astype(np.float32)
    w = rng.dirichlet(np.ones(C))
    return dict(means=means, log_weights=np.log(w).astype(np.float32),
                comp_var=float(cfg["comp_var"]))


def bytes_per_element(dtype):
    return 2 if dtype == "bf16" else 4


def main_pass_bytes(B, L, d, dtype):
    """Algorithmic bytes of the log-ratio pass: x, m^q, m^p read once."""
    return 3 * B * L * d * bytes_per_element(dtype)


def describe(kind):
    c = VERIFY_CONFIGS[kind]
    return "%s: B=%d L=%d d=%d %s" % (kind, c["B"], c["L"], c["d"], c["dtype"])


__all__ = ["VERIFY_CONFIGS", "SAMPLER_CONFIG", "sigma_schedule", "round_to_bf16",
           "make_verify_inputs", "make_gmm", "main_pass_bytes", "describe", "math"]
