"""sdv_verify_pipelined: runs of independent verification calls whose kernels may overlap
on one stream (each call streams its window while the previous call's chains finish).

A pipelined call streams with the same tile reduction as a plain call, so its log
ratios, accepted lengths and status bits equal a plain call's bit for bit; it finishes
every chain with k_finish (the one-warp U-sampler, a 64-thread residual writer), so its
U and states agree with a plain call's within the parity tolerances (U: 5e-6 + 3e-7|U|;
states: 1e-5 absolute for fp32, 2e-2 for bf16), and one run is compared with the oracle
directly.  Checked with separate outputs per call, with outputs shared by all calls
(written in call order), under CUDA-graph capture, and with one workspace of arbitrary
contents reused by calls of changing sizes."""
import numpy as np
import pytest
import torch

import workloads as W
from gpu_helpers import compare, oracle_for, to_dev
from oracle import verify as OV

pytestmark = pytest.mark.gpu

KEYS = ("accepted_len", "y", "status", "log_ratio", "delta_norm", "aux")


@pytest.fixture(scope="module")
def api():
    import __graft_entry__ as g
    g.build()
    from paper_2606_13426_gb300 import api as A
    return A


def _sets(kind, n, B, L, d, ragged):
    out = []
    for i in range(n):
        inp = W.make_verify_inputs(kind, B=B, L=L, d=d, seed=50 + i, per_chain_sigma=True)
        s = dict(x=to_dev(inp, "x_draft"), mq=to_dev(inp, "mu_target"), mp=to_dev(inp, "mu_draft"),
                 sigma=torch.from_numpy(inp["sigma"]).cuda())
        if ragged:
            rng = np.random.Generator(np.random.PCG64(60 + i))
            Leff = rng.integers(0, L + 1, B).astype(np.int32)
            Leff[:2] = [0, L]
            s["L_eff"] = torch.from_numpy(Leff).cuda()
            s["mu_target_bonus"] = torch.from_numpy(rng.standard_normal((B, d)).astype(np.float32)).cuda().to(s["x"].dtype)
            s["sigma_bonus"] = torch.from_numpy(rng.uniform(0.1, 1.0, B).astype(np.float32)).cuda()
        out.append(s)
    return out


def _call(api, s, seed, mode, ws, out=None, pipelined=False):
    kw = {k: s[k] for k in ("L_eff", "mu_target_bonus", "sigma_bonus") if k in s}
    return api.verify(s["x"], s["mq"], s["mp"], s["sigma"], seed, mode, with_aux=True, workspace=ws,
                      out=out, pipelined=pipelined, **kw)


TOL_Y = {torch.float32: 1e-5, torch.bfloat16: 2e-2}


def _same(a, b, mask=None):
    """a (pipelined) against b (plain call on the same inputs)."""
    for k in ("accepted_len", "log_ratio", "delta_norm"):
        assert torch.equal(a[k], b[k]), k
    m = torch.ones(a["y"].shape[0], dtype=torch.bool, device=a["y"].device) if mask is None else mask
    assert torch.equal(a["status"][m], b["status"][m])
    yb = b["y"][m].float()
    err = (a["y"][m].float() - yb).abs()
    if a["y"].dtype == torch.bfloat16:      # both rounded to bf16: one ulp of the output apart at most
        tol = torch.clamp(2.0 ** -7 * yb.abs(), min=TOL_Y[torch.bfloat16])
    else:
        tol = torch.full_like(yb, TOL_Y[torch.float32])
    assert err.numel() == 0 or bool(torch.all(err <= tol)), err.max().item()
    ua, ub = a["aux"][m, 0], b["aux"][m, 0]
    fin = torch.isfinite(ub)
    assert torch.equal(torch.isfinite(ua), fin)
    assert torch.all((ua[fin] - ub[fin]).abs() <= 5e-6 + 3e-7 * ub[fin].abs())


CASES = [("pixel", 64, 8, 3072, False), ("latent", 16, 16, 16384, False), ("pixel", 40, 6, 1000, True),
         ("tiny", 8, 4, 37, True)]


@pytest.mark.parametrize("kind,B,L,d,ragged", CASES)
@pytest.mark.parametrize("mode", ["block", "sample"])
def test_pipelined_calls_equal_plain_calls(api, kind, B, L, d, ragged, mode):
    sets = _sets(kind, 4, B, L, d, ragged)
    dt = sets[0]["x"].dtype
    ws = torch.zeros(api.workspace_bytes(B, L, d, dt), dtype=torch.uint8, device="cuda")
    n = 12
    torch.cuda.synchronize()
    piped = [_call(api, sets[i % 4], 100 + i, mode, ws, pipelined=True) for i in range(n)]
    torch.cuda.synchronize()
    for i in range(n):
        ref = _call(api, sets[i % 4], 100 + i, mode, ws)
        act = torch.ones(B, dtype=torch.bool, device="cuda") if not ragged else sets[i % 4]["L_eff"] > 0
        _same(piped[i], ref, act)
    # the last pipelined call against the oracle
    inp = W.make_verify_inputs(kind, B=B, L=L, d=d, seed=50 + (n - 1) % 4, per_chain_sigma=True)
    kw = {}
    if ragged:
        st = sets[(n - 1) % 4]
        kw = dict(Leff=st["L_eff"].cpu().numpy(), mu_target_bonus=st["mu_target_bonus"].float().cpu().numpy(),
                  sigma_bonus=st["sigma_bonus"].cpu().numpy())
    m = OV.MODE_BLOCK if mode == "block" else OV.MODE_SAMPLE
    o = oracle_for(inp, 100 + n - 1, m, **kw)
    g = {k: (v.float().cpu().numpy() if v.dtype == torch.bfloat16 else v.cpu().numpy())
         for k, v in piped[n - 1].items()}
    compare(g, o, m, inp["dtype"])


@pytest.mark.parametrize("kind,B,L,d,ragged", CASES[:2])
def test_pipelined_calls_sharing_outputs(api, kind, B, L, d, ragged):
    """Every call writes the same output buffers; they end with the last call's outputs."""
    sets = _sets(kind, 3, B, L, d, ragged)
    dt = sets[0]["x"].dtype
    ws = torch.zeros(api.workspace_bytes(B, L, d, dt), dtype=torch.uint8, device="cuda")
    out = {}
    first = _call(api, sets[0], 7, "block", ws, out=out, pipelined=True)
    out.update(first)
    for i in range(1, 10):
        r = _call(api, sets[i % 3], 7 + i, "block", ws, out=out, pipelined=True)
    torch.cuda.synchronize()
    ref = _call(api, sets[9 % 3], 16, "block", ws)
    _same(r, ref)


def test_pipelined_calls_in_a_cuda_graph(api):
    kind, B, L, d = "pixel", 96, 8, 3072
    sets = _sets(kind, 4, B, L, d, False)
    ws = torch.zeros(api.workspace_bytes(B, L, d, torch.float32), dtype=torch.uint8, device="cuda")
    outs = [dict(accepted_len=torch.empty(B, dtype=torch.int32, device="cuda"),
                 y=torch.empty(B, d, device="cuda"), status=torch.empty(B, dtype=torch.int32, device="cuda"),
                 log_ratio=torch.empty(B, L, device="cuda"), delta_norm=torch.empty(B, L, device="cuda"),
                 aux=torch.empty(B, 4, device="cuda")) for _ in range(8)]
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        _call(api, sets[0], 1, "block", ws)          # warm-up outside capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(8):
            _call(api, sets[i % 4], 300 + i, "block", ws, out=outs[i], pipelined=True)
    for _ in range(2):
        for o in outs:
            for v in o.values():
                v.fill_(-7)
        g.replay()
        torch.cuda.synchronize()
        for i in range(8):
            _same(outs[i], _call(api, sets[i % 4], 300 + i, "block", ws))


def test_pipelined_long_rows(api):
    """Rows longer than 16384 elements: k_tiles + k_finish without the residual, then the
    long-row residual kernels, all four launched to overlap their predecessors (the
    residual kernels sit resident, few and long, while the next call streams).  Against
    plain calls on the same inputs (ratios, tau and status exact; U and states within
    the parity tolerance), with separate outputs, and the last call against the oracle."""
    B, L, d = 3, 4, 16388
    sets = _sets("pixel", 2, B, L, d, False)
    ws = torch.zeros(api.workspace_bytes(B, L, d, torch.float32), dtype=torch.uint8, device="cuda")
    piped = [_call(api, sets[i % 2], 500 + i, "block", ws, pipelined=True) for i in range(6)]
    torch.cuda.synchronize()
    for i in range(6):
        _same(piped[i], _call(api, sets[i % 2], 500 + i, "block", ws))
    inp = W.make_verify_inputs("pixel", B=B, L=L, d=d, seed=50 + 5 % 2, per_chain_sigma=True)
    o = oracle_for(inp, 505, OV.MODE_BLOCK)
    g = {k: v.cpu().numpy() for k, v in piped[5].items()}
    compare(g, o, OV.MODE_BLOCK, "f32")


def test_pipelined_long_rows_many_chains(api):
    """Many chains with long rows: the residual kernels keep one chunk per chain at least
    (more chains than their CTA budget)."""
    B, L, d = 520, 2, 16388
    sets = _sets("pixel", 1, B, L, d, False)
    ws = torch.zeros(api.workspace_bytes(B, L, d, torch.float32), dtype=torch.uint8, device="cuda")
    piped = [_call(api, sets[0], 700 + i, "sample", ws, pipelined=True) for i in range(2)]
    torch.cuda.synchronize()
    for i in range(2):
        _same(piped[i], _call(api, sets[0], 700 + i, "sample", ws))


def test_pipelined_calls_reuse_a_workspace_across_sizes(api):
    """One workspace of arbitrary contents (filled with 0xFF bytes) serves a run of
    pipelined calls whose sizes change from call to call, so that each call's tile
    partials land on slots that a call of other sizes left behind: the partials' tags
    keep every call to its own (against plain calls on a fresh workspace)."""
    shapes = [(64, 8, 3072), (160, 4, 1000), (96, 8, 3072), (72, 6, 2048), (200, 2, 520)]
    sets = {sh: _sets("pixel", 1, *sh, False)[0] for sh in shapes}
    nbytes = max(api.workspace_bytes(B, L, d, torch.float32) for B, L, d in shapes)
    ws = torch.full((nbytes,), 255, dtype=torch.uint8, device="cuda")
    order = shapes + shapes[::-1] + shapes
    piped = [_call(api, sets[sh], 900 + i, "block", ws, pipelined=True) for i, sh in enumerate(order)]
    torch.cuda.synchronize()
    for i, sh in enumerate(order):
        fresh = torch.zeros(api.workspace_bytes(*sh, torch.float32), dtype=torch.uint8, device="cuda")
        _same(piped[i], _call(api, sets[sh], 900 + i, "block", fresh))
