"""Benchmark of the speculative-diffusion verification step on GB300.

One step = one verification call (sdv_verify_pipelined: k_tiles streams the window and
reduces the log-ratio partials, k_finish runs the acceptance rule, the residual U-draw
and the residual write) on one batch of the pixel-scale workload (B=256 chains, L=8 draft steps, d=3x32x32 fp32, block
verification) with inputs resident in HBM.  Eight input sets (8 x 75.5 MB, well
above the 129 MB L2) rotate between steps, so every step reads its inputs from HBM.
Steps are independent batches of chains: consecutive calls may overlap on the GPU (a
call streams its window while the previous call's last chains finish).  Steps are
captured into CUDA graphs and replayed.

Prints ONE JSON line (rank 0):
  value        verified draft-steps/s (B*L per step), whole job
  roofline     full-call algorithmic bytes per call / the per-call period of 200
               back-to-back calls in one graph (events at its two ends only), vs the
               measured HBM copy peak
  steady_state the per-call period over >= 1 s of replays of the timed graph
  workloads    the same figures for the latent (bf16) and high-resolution workloads,
               and the end-to-end sampler's wall-clock
  e2e          the same metric through the public API from pinned host memory
               (api.HostStream: window copied in, results copied out, every step)
  cpu_baseline the CPU oracle on a bounded sample of the same workload

--impl reference times the CPU oracle alone (the reference arm of this build).
"""
import argparse
import hashlib
import json
import math
import os
import re
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import workloads as W  # noqa: E402

METRIC = "verified draft-steps/s and HBM GB/s vs ~8 TB/s; mean accepted steps/target call"
UNIT = "draft-steps/s"
N_SETS = 8


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=2000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default="pixel", choices=["pixel", "latent", "highres", "sampler"])
    p.add_argument("--sampler-L", default="4,8,16",
                   help="draft windows of the end-to-end sampler workload")
    p.add_argument("--sampler-rounds", type=int, default=0,
                   help="sampler workload only: instead of the timed runs, drive this many "
                        "rounds from the host (sdv_sampler_begin / _round / _end, block mode), "
                        "twice per window, so that a profiler sees every kernel launch")
    p.add_argument("--mode", default="block", choices=["block", "sample"])
    p.add_argument("--batch", type=int, default=0,
                   help="chains per call (0: the workload's B); smaller batches serve ncu captures")
    p.add_argument("--no-pipeline", action="store_true",
                   help="time sdv_verify_ex calls instead of sdv_verify_pipelined")
    p.add_argument("--headline-only", action="store_true",
                   help="skip the latent / high-resolution / sampler sub-results")
    p.add_argument("--profile", action="store_true",
                   help="profiler runs: the warm-up and timed steps of the headline workload only "
                        "(no 200-call pass, steady state, e2e, tau statistics or CPU baseline)")
    p.add_argument("--cpu-seconds", type=float, default=12.0)
    p.add_argument("--skip-cpu", action="store_true")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


def kernel_sources_digest():
    """sha256 over the sources that define the fused verify kernel (in a fixed order)."""
    h = hashlib.sha256()
    for f in ("sdv_verify.cu", "sdv_device.cuh", "sdv_host.h"):
        with open(os.path.join(ROOT, "paper_2606_13426_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def profile_traffic(workload, full_size, pipelined=True):
    """DRAM bytes per call (all of the call's kernels) on this workload from its committed
    ncu summary (profiles/verify_<workload>_<pipelined|plain>.md), if the kernel sources
    are unchanged since the capture and the batch is the workload's full one (else None)."""
    path = os.path.join(ROOT, "profiles", "verify_%s_%s.md" % (workload, "pipelined" if pipelined else "plain"))
    if not full_size or not os.path.exists(path):
        return None
    txt = open(path).read()
    m = re.search(r"traffic_bytes_per_call:\s*([0-9.eE+]+)", txt)
    h = re.search(r"kernel_source_sha256:\s*([0-9a-f]+)", txt)
    if not m or not h:
        return None
    return float(m.group(1)) if h.group(1) == kernel_sources_digest() else None


class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = [r.split(",") for r in out.strip().splitlines() if r.strip()]
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, r[5:9]):
                if v.strip().lower() in ("active", "1", "yes"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": float(np.median(sm)), "sm_max_mhz": float(max(mx)),
                "reasons": sorted(reasons), "samples": len(sm)}


# Rows of more than this many groups of four elements get their residual from two
# extra kernels (the library's kFusedMaxGroups and kFinishMaxGroups); pipelined calls
# keep rows of up to PIPE_MAX_GROUPS in k_finish (kPipeMaxGroups).
FUSED_MAX_GROUPS = 1024
FINISH_MAX_GROUPS = 1024
PIPE_MAX_GROUPS = 4096

# From this many chains on, the library streams the tiles with k_tiles and finishes
# every chain with one warp of k_finish (the library's kManyChainMin).
MANY_CHAIN_MIN = 512


def many_chains(B):
    return B >= MANY_CHAIN_MIN


def pipelined_path(d, pipelined):
    """Does the call take the pipelined path (every kernel launched to overlap its
    predecessor)?  Every pipelined call does."""
    return bool(pipelined)


def wide_finish(B, d, pipelined=False):
    """Rows of 1025-4096 groups of four finished by a 256-thread k_finish (pipelined
    calls, or plain calls with fewer than MANY_CHAIN_MIN chains)."""
    ng = (d + 3) // 4
    return FINISH_MAX_GROUPS < ng <= PIPE_MAX_GROUPS and (pipelined or not many_chains(B))


# Plain calls with fewer chains run the fused kernel (the library's kFusedMaxChains).
FUSED_MAX_CHAINS = 64


def _two_kernels(B, d, pipelined):
    return B >= FUSED_MAX_CHAINS or bool(pipelined) or wide_finish(B, d, pipelined)


def long_rows(d, B=0, pipelined=False):
    """Rows whose residual two extra kernels write (longer than the finishing CTA's noise
    cache: the fused kernel's, or k_finish's)."""
    if wide_finish(B, d, pipelined):
        return False
    return (d + 3) // 4 > (FINISH_MAX_GROUPS if _two_kernels(B, d, pipelined) else FUSED_MAX_GROUPS)


def launches_per_step(B, d, pipelined=False):
    """Kernels one verification call launches: the fused verify kernel, or k_tiles and
    k_finish (many chains, a pipelined call, or rows of 1025-4096 groups), plus the
    residual dot / write kernels for long rows."""
    return (2 if _two_kernels(B, d, pipelined) else 1) + (2 if long_rows(d, B, pipelined) else 0)


def kernels_of_step(B, d, pipelined=False):
    names = ["k_tiles", "k_finish"] if _two_kernels(B, d, pipelined) else ["k_verify"]
    if long_rows(d, B, pipelined):
        names += ["k_resid_dot", "k_resid_write"]
    return names


def call_bytes(B, L, d, dtype):
    """Algorithmic bytes of one call: x, m^q, m^p read once, and the residual pass: the
    rejected row's m^q and m^p re-read plus y written (upper bound: every chain)."""
    s = W.bytes_per_element(dtype)
    return 3 * B * L * d * s + 3 * B * d * s


def input_seed(base, i, rank):
    """Seed of input set i on this rank: every rank verifies its own chains (weak scaling,
    no data-path collective)."""
    return base + 100 * i + 7 * rank


def max_over_ranks(x, pg, device):
    """The largest of the ranks' values of x (the job's time is its slowest rank's)."""
    if pg is None:
        return float(x)
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    pg.all_reduce(t, op=pg.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world, units_per_rank, seconds):
    """Units processed by all ranks per second of the slowest rank."""
    return world * units_per_rank / seconds


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def cpu_oracle_rate(inp, seed, mode, seconds, max_chains=None):
    """Time oracle.verify on whole-chain samples of one input set until ~seconds elapse."""
    from oracle import verify as OV
    m = OV.MODE_BLOCK if mode == "block" else OV.MODE_SAMPLE
    Bn, L = inp["B"], inp["L"]
    chains_done, t_total, calls = 0, 0.0, 0
    per_call = Bn if max_chains is None else min(Bn, max_chains)
    rng = np.random.Generator(np.random.PCG64(0))
    while t_total < seconds:
        ch = np.sort(rng.choice(Bn, per_call, replace=False))
        t0 = time.perf_counter()
        OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], seed + calls,
                  m, chains=ch)
        t_total += time.perf_counter() - t0
        chains_done += per_call
        calls += 1
    return chains_done * L / t_total, chains_done, t_total


def _oracle_worker(job):
    """One process of the all-cores oracle timing: the same input set, its own chains."""
    workload, Bn, seed, mode, seconds, wid, nw, barrier = job
    from oracle import verify as OV
    inp = W.make_verify_inputs(workload, B=Bn, seed=seed)
    m = OV.MODE_BLOCK if mode == "block" else OV.MODE_SAMPLE
    own = np.arange(wid, Bn, nw)
    barrier.wait()
    chains_done, t_total, calls = 0, 0.0, 0
    while t_total < seconds:
        t0 = time.perf_counter()
        OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], 1000 * wid + calls,
                  m, chains=own)
        t_total += time.perf_counter() - t0
        chains_done += len(own)
        calls += 1
    return chains_done, t_total


def cpu_oracle_rate_all_cores(workload, Bn, seed, mode, seconds, nproc):
    """The oracle as it stands in nproc spawned processes (one thread each), each on its
    own share of the chains of the same input set, started together."""
    import multiprocessing as mpl
    ctx = mpl.get_context("spawn")
    with ctx.Manager() as mgr:
        barrier = mgr.Barrier(nproc)
        with ctx.Pool(nproc) as pool:
            res = pool.map(_oracle_worker, [(workload, Bn, seed, mode, seconds, w, nproc, barrier)
                                            for w in range(nproc)])
    chains = sum(r[0] for r in res)
    t = max(r[1] for r in res)
    L = W.VERIFY_CONFIGS[workload]["L"]
    return chains * L / t, chains, t


def workload_name(args, Bn, L, d, dt_name):
    """config.workload of a verify run, identical in both arms."""
    return "%s verify (B=%d, L=%d, d=%d %s), %s mode" % (args.workload, Bn, L, d, dt_name, args.mode)


def run_reference(args, world, rank):
    """Reference arm: the CPU oracle as it stands, on the host cores, same workload/metric."""
    if rank != 0:
        return
    cfg = W.VERIFY_CONFIGS[args.workload]
    inp = W.make_verify_inputs(args.workload)
    from oracle import verify as OV
    m = OV.MODE_BLOCK if args.mode == "block" else OV.MODE_SAMPLE
    # calibrate: chains per step so that warmup + steps take ~120 s at most
    t0 = time.perf_counter()
    OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], 0, m,
              chains=np.arange(1))
    t1 = time.perf_counter() - t0
    budget = 120.0 / max(1, args.steps + args.warmup)
    per_step = int(max(1, min(cfg["B"], budget / max(t1, 1e-6))))
    rng = np.random.Generator(np.random.PCG64(1))
    for w in range(args.warmup):
        OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], w, m,
                  chains=rng.choice(cfg["B"], per_step, replace=False))
    t0 = time.perf_counter()
    for s in range(args.steps):
        OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], 1000 + s, m,
                  chains=rng.choice(cfg["B"], per_step, replace=False))
    dt = time.perf_counter() - t0
    value = args.steps * per_step * cfg["L"] / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": workload_name(args, cfg["B"], cfg["L"], cfg["d"], cfg["dtype"]),
                   "global_batch": cfg["B"], "window": cfg["L"], "dim": cfg["d"],
                   "parallelism": "host, one thread"},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": "%d chain(s) of the %s batch per step (oracle.verify, numpy fp64)"
                                   % (per_step, args.workload)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line))


def run_sampler_rounds(args, rank, local):
    """Host-driven sampler rounds (profiling aid): per window L, two runs of
    begin + R rounds + end in block mode; prints the time per round of the second."""
    import torch
    import __graft_entry__ as G
    G.build()
    from paper_2606_13426_gb300 import api
    torch.cuda.set_device(local)
    cfg = W.SAMPLER_CONFIG
    gm = W.make_gmm()
    tgt = api.GmmTarget(torch.from_numpy(gm["means"]), torch.from_numpy(gm["log_weights"]),
                        gm["comp_var"], cfg["K"], cfg["churn"])
    Bn, d, R = cfg["B"], cfg["d"], args.sampler_rounds
    runs = {}
    for L in [int(v) for v in args.sampler_L.split(",")]:
        ws = torch.empty(api.B.sdv_sampler_workspace_bytes(Bn, L, d), dtype=torch.uint8, device="cuda")
        for _ in range(2):
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            r = api.sampler_rounds(Bn, L, tgt, 100, R, "block", workspace=ws)
            torch.cuda.synchronize()
            t = time.perf_counter() - t0
        runs["L%d_block" % L] = {"rounds": r["rounds"], "us_per_round": 1e6 * t / max(1, R)}
    if rank == 0:
        print(json.dumps({"metric": "host-driven sampler rounds (profiling aid, not a bench value)",
                          "config": {"B": Bn, "d": d, "rounds": R}, "runs": runs}))


def cpu_sampler_rates(n_chains, L=4, mode="block"):
    """The oracle sampler and the oracle's plain Euler-Maruyama chain on the first
    n_chains chains of the sampler workload (one thread): denoising steps/s of each."""
    from oracle import sampler as OS
    from oracle import verify as OV
    cfg = W.SAMPLER_CONFIG
    gm = W.make_gmm()
    sch = OS.VPSchedule(cfg["K"], cfg["churn"], cfg["beta_min"], cfg["beta_max"], cfg["t_floor"])
    chains = np.arange(n_chains)
    m = OV.MODE_BLOCK if mode == "block" else OV.MODE_SAMPLE
    t0 = time.perf_counter()
    OS.speculative_sample(cfg["B"], cfg["d"], L, m, gm, sch, seed=100, chains=chains)
    t_spec = time.perf_counter() - t0
    t0 = time.perf_counter()
    OS.em_sample(cfg["B"], cfg["d"], gm, sch, 1, chains=chains)
    t_em = time.perf_counter() - t0
    return n_chains * cfg["K"] / t_spec, n_chains * cfg["K"] / t_em, t_spec, t_em


def run_sampler(args, world, rank, local):
    """End-to-end speculative sampler on the analytic 8-component mixture (B = 1024 chains,
    d = 1024, K = 1000 VP Euler-Maruyama steps, churn 0.5, Free and Frozen drafters)
    against the plain Euler-Maruyama chain: wall-clock, rounds and accepted steps per
    parallel target call (the Frozen drafter makes one more target call per round)."""
    import torch
    import __graft_entry__ as G
    G.build()
    from paper_2606_13426_gb300 import api
    torch.cuda.set_device(local)
    cfg = W.SAMPLER_CONFIG
    gm = W.make_gmm()
    tgt = api.GmmTarget(torch.from_numpy(gm["means"]), torch.from_numpy(gm["log_weights"]),
                        gm["comp_var"], cfg["K"], cfg["churn"])
    Bn, d, K = cfg["B"], cfg["d"], cfg["K"]

    def timed(fn):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out = fn()
        torch.cuda.synchronize()
        return out, time.perf_counter() - t0

    timed(lambda: api.em_sample(Bn, tgt, 1))
    t_em = min(timed(lambda: api.em_sample(Bn, tgt, 1 + i))[1] for i in range(3))
    runs = {}
    for L in [int(v) for v in args.sampler_L.split(",")]:
        ws = torch.empty(api.B.sdv_sampler_workspace_bytes(Bn, L, d), dtype=torch.uint8, device="cuda")
        for drafter in ("free", "frozen"):
            for mode in ("sample", "block"):
                timed(lambda: api.sampler_run(Bn, L, tgt, 7, mode, drafter, workspace=ws))
                best = None
                for i in range(3):
                    r, t = timed(lambda: api.sampler_run(Bn, L, tgt, 100 + i, mode, drafter, workspace=ws))
                    if best is None or t < best[1]:
                        best = (r, t)
                r, t = best
                cr = r["chain_rounds"].cpu().numpy().astype(np.float64)
                ts = r["tau_sum"].cpu().numpy().astype(np.float64)
                calls_per_round = 2.0 if drafter == "frozen" else 1.0
                runs["L%d_%s%s" % (L, mode, "_frozen" if drafter == "frozen" else "")] = {
                    "ms": 1e3 * t, "rounds": r["rounds"], "mean_chain_rounds": float(cr.mean()),
                    "mean_tau": float(ts.sum() / cr.sum()),
                    "target_calls_per_chain": float(calls_per_round * cr.mean() + 1.0),
                    "speedup_vs_em": t_em / t}
    best_key = min(runs, key=lambda k2: runs[k2]["ms"])
    line = {
        "metric": "end-to-end speculative sampler: denoising steps/s; mean accepted steps/target call",
        "value": Bn * K / (runs[best_key]["ms"] * 1e-3), "unit": "denoising steps/s",
        "n_gpus": 1, "higher_is_better": True, "dtype": "f32", "data": "synthetic",
        "config": {"workload": "analytic 8-component GMM, d=%d, B=%d, K=%d VP EM steps, churn %.2f, "
                               "Free and Frozen drafters" % (d, Bn, K, cfg["churn"]), "best": best_key},
        "em_ms": 1e3 * t_em, "em_steps_per_s": Bn * K / t_em, "runs": runs,
    }
    if rank == 0 and not args.skip_cpu:
        n_cpu = 8
        spec_rate, em_rate, t_spec, t_em_cpu = cpu_sampler_rates(n_cpu)
        line["cpu_baseline"] = {
            "value": spec_rate, "unit": "denoising steps/s", "cores": 1, "kind": "oracle",
            "sample": "%d of the %d chains through oracle.sampler.speculative_sample (L=4, block, "
                      "Free drafter; numpy fp64, one thread), %.1f s; the oracle's plain EM chain on "
                      "the same chains: %.4g denoising steps/s (%.1f s)" % (n_cpu, Bn, t_spec, em_rate, t_em_cpu)}
    if rank == 0:
        print(json.dumps(line))


def _graph_of_calls(stream, n, call):
    """A CUDA graph of n calls call(0..n-1) captured on `stream`."""
    import torch
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for i in range(n):
            call(i)
    return g


def _replay_ms(stream, graphs, reps=1):
    """Device time of replaying `graphs` (in order, `reps` times) between two events."""
    import torch
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(reps):
            for g in graphs:
                g.replay()
        e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1)


def measure_verify(api, name, Bn, mode, steps, warmup, dev, rank, pg=None, clocks=None, pipelined=True,
                   profile=False):
    """Timed verification calls on workload `name`: the timed region (steps calls in CUDA
    graph replays, events at its ends), the per-call period of 200 back-to-back calls
    (the roofline's duration), the steady-state period over >= 1 s of replays, and mean
    tau per target call in both modes.  Returns a dict; the input sets stay on the device
    only while it runs."""
    import torch
    cfg = W.VERIFY_CONFIGS[name]
    L, d, dt_name = cfg["L"], cfg["d"], cfg["dtype"]
    tdt = torch.bfloat16 if dt_name == "bf16" else torch.float32
    set_bytes = W.main_pass_bytes(Bn, L, d, dt_name)
    props = torch.cuda.get_device_properties(dev)
    l2 = getattr(props, "L2_cache_size", 129 * 2 ** 20)
    n_sets = max(1, min(N_SETS, math.ceil(4 * l2 / set_bytes))) if set_bytes < 4 * l2 else 1

    def to_dev(inp, key):
        if dt_name == "bf16":
            return torch.from_numpy(inp[key + "_bits"].view(np.int16)).to(dev).view(torch.bfloat16)
        return torch.from_numpy(inp[key]).to(dev)

    sets, host0 = [], None
    for i in range(n_sets):
        inp = W.make_verify_inputs(name, B=Bn, seed=input_seed(cfg["seed"], i, rank))
        sets.append(dict(x=to_dev(inp, "x_draft"), mq=to_dev(inp, "mu_target"),
                         mp=to_dev(inp, "mu_draft"), sigma=torch.from_numpy(inp["sigma"]).to(dev)))
        if i == 0:
            host0 = inp
    outs = dict(accepted_len=torch.empty(Bn, dtype=torch.int32, device=dev),
                y=torch.empty(Bn, d, dtype=tdt, device=dev),
                status=torch.empty(Bn, dtype=torch.int32, device=dev))
    ws = torch.zeros(max(api.workspace_bytes(Bn, L, d, tdt), 256), dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step(i, m=mode):
        st = sets[i % n_sets]
        api.verify(st["x"], st["mq"], st["mp"], st["sigma"], seed=i, mode=m, with_ratios=False,
                   workspace=ws, out=outs, pipelined=pipelined)

    with torch.cuda.stream(stream):
        for i in range(max(warmup, 1)):
            step(i)
    torch.cuda.synchronize()
    g_steps = min(steps, 256)
    reps, rem = divmod(steps, g_steps)
    g_main = _graph_of_calls(stream, g_steps, step)
    graphs = [g_main] * reps
    if rem:
        graphs.append(_graph_of_calls(stream, rem, step))
    _replay_ms(stream, graphs[:1])                            # graph warm-up

    if pg:
        pg.barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
        time.sleep(0.3)
    ms_total = _replay_ms(stream, graphs)
    ms_total = max_over_ranks(ms_total, pg, dev)
    if pg:
        pg.barrier()
    ms_step = ms_total / steps
    if profile:
        clk = clocks.stop() if clocks else None
        return dict(name=name, ms_step=ms_step, clocks=clk)

    # the roofline's duration: 200 back-to-back calls in one graph, events at its ends only
    g200 = _graph_of_calls(stream, 200, step)
    _replay_ms(stream, [g200])
    ms_call = min(_replay_ms(stream, [g200]) for _ in range(3)) / 200
    # steady state: replays of the 200-call graph for >= 1 s (clocks sampled throughout)
    reps_ss = max(1, int(math.ceil(1000.0 / max(ms_call * 200, 1e-3))))
    ms_ss = _replay_ms(stream, [g200], reps=reps_ss) / (200 * reps_ss)
    clk = clocks.stop() if clocks else None

    taus = {}
    for m in ("block", "sample"):
        acc = []
        for i, st in enumerate(sets):
            r = api.verify(st["x"], st["mq"], st["mp"], st["sigma"], seed=10_000 + i, mode=m,
                           with_ratios=False, workspace=ws)
            acc.append(r["accepted_len"].cpu().numpy())
        taus[m] = float(np.concatenate(acc).mean() + 1.0)
    del sets, g_main, graphs, g200
    torch.cuda.synchronize()
    torch.cuda.empty_cache()

    hbm_peak, peak_kind = peaks()
    nbytes = call_bytes(Bn, L, d, dt_name)
    achieved = nbytes / (ms_call * 1e-3) / 1e9
    return dict(
        name=name, B=Bn, L=L, d=d, dtype=dt_name, n_sets=n_sets, set_bytes=set_bytes, l2=l2,
        ms_step=ms_step, ms_call=ms_call, ms_steady=ms_ss, steady_calls=200 * reps_ss,
        value_per_rank=Bn * L / (ms_step * 1e-3), taus=taus, clocks=clk, host0=host0,
        roofline={"bound": "hbm", "achieved": achieved, "peak": hbm_peak, "unit": "GB/s",
                  "frac": achieved / hbm_peak, "peak_kind": peak_kind,
                  "kernel": ("k_verify (fused: log-ratio pass, acceptance, U-draw, residual write)"
                             if launches_per_step(Bn, d, pipelined) == 1 else
                             "whole call (%d kernels: %s)" % (launches_per_step(Bn, d, pipelined),
                                                             ", ".join(kernels_of_step(Bn, d, pipelined)))),
                  "duration": "per-call period of 200 back-to-back calls in one CUDA graph "
                              "(events at its two ends only)",
                  "duration_us": 1e3 * ms_call, "algorithmic_bytes": nbytes,
                  "traffic": profile_traffic(name, Bn == cfg["B"], pipelined_path(d, pipelined))})


def measure_e2e(api, host0, Bn, L, d, dt_name, mode, dev, n_steps):
    """The metric through the public API from pinned host memory: api.HostStream copies
    each step's window in (one [3, B, L, d] copy) while the previous step verifies, and
    copies its accepted lengths and states back; timed on the host clock."""
    import torch
    tdt = torch.bfloat16 if dt_name == "bf16" else torch.float32
    win = torch.empty(3, Bn, L, d, dtype=tdt, pin_memory=True)
    for k, key in enumerate(("x_draft", "mu_target", "mu_draft")):
        if dt_name == "bf16":
            win[k].view(torch.int16).copy_(torch.from_numpy(host0[key + "_bits"].view(np.int16)))
        else:
            win[k].copy_(torch.from_numpy(host0[key]))
    sig = torch.from_numpy(host0["sigma"]).pin_memory()
    hs = api.HostStream(Bn, L, d, tdt, tuple(sig.shape), depth=2, device=dev)
    for i in range(4):
        hs.result(hs.submit(win, sig, i, mode))
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    prev = None
    for i in range(n_steps):
        cur = hs.submit(win, sig, i, mode)
        if prev is not None:
            hs.result(prev)
        prev = cur
    hs.result(prev)
    e2e_s = (time.perf_counter() - t0) / n_steps
    h2d = win.numel() * win.element_size() + sig.numel() * 4
    d2h = Bn * 4 + Bn * d * win.element_size()
    return e2e_s, h2d, d2h


def sampler_summary(api, dev):
    """Wall-clock of the end-to-end sampler (L = 8, block, Free drafter; best of three)
    against the plain Euler-Maruyama chain, on the sampler workload."""
    import torch
    cfg = W.SAMPLER_CONFIG
    gm = W.make_gmm()
    tgt = api.GmmTarget(torch.from_numpy(gm["means"]), torch.from_numpy(gm["log_weights"]),
                        gm["comp_var"], cfg["K"], cfg["churn"], device=dev)
    Bn, d, K, L = cfg["B"], cfg["d"], cfg["K"], 8

    def timed(fn):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        out = fn()
        torch.cuda.synchronize()
        return out, time.perf_counter() - t0

    timed(lambda: api.em_sample(Bn, tgt, 1))
    t_em = min(timed(lambda: api.em_sample(Bn, tgt, 2 + i))[1] for i in range(3))
    ws = torch.empty(api.B.sdv_sampler_workspace_bytes(Bn, L, d), dtype=torch.uint8, device=dev)
    timed(lambda: api.sampler_run(Bn, L, tgt, 7, "block", "free", workspace=ws))
    best = min((timed(lambda: api.sampler_run(Bn, L, tgt, 100 + i, "block", "free", workspace=ws))
                for i in range(3)), key=lambda rt: rt[1])
    r, t = best
    cr = r["chain_rounds"].cpu().numpy().astype(np.float64)
    ts = r["tau_sum"].cpu().numpy().astype(np.float64)
    return {"workload": "analytic 8-component GMM, d=%d, B=%d, K=%d, L=%d, block, Free drafter"
                        % (d, Bn, K, L),
            "ms": 1e3 * t, "rounds": r["rounds"], "mean_tau": float(ts.sum() / cr.sum()),
            "denoising_steps_per_s": Bn * K / t, "em_ms": 1e3 * t_em}


def main():
    args = parse()
    world, rank, local = dist_setup()
    if args.impl == "reference":
        run_reference(args, world, rank)
        return
    if args.workload == "sampler" and args.sampler_rounds > 0:
        run_sampler_rounds(args, rank, local)
        return
    if args.workload == "sampler":
        run_sampler(args, world, rank, local)
        return

    import torch
    import __graft_entry__ as G
    G.build()
    from paper_2606_13426_gb300 import api

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    pg = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
        pg = dist

    cfg = W.VERIFY_CONFIGS[args.workload]
    Bn = args.batch if args.batch > 0 else cfg["B"]
    L, d, dt_name = cfg["L"], cfg["d"], cfg["dtype"]
    pipelined = not args.no_pipeline
    clocks = ClockSampler(local)
    head = measure_verify(api, args.workload, Bn, args.mode, args.steps, args.warmup, dev, rank, pg,
                          clocks, pipelined, profile=args.profile)
    value = whole_job_rate(world, Bn * L, head["ms_step"] * 1e-3)
    if args.profile:
        if rank == 0:
            print(json.dumps({"metric": "profiler run (not a bench value)", "ms_per_step": head["ms_step"],
                              "steps": args.steps, "workload": args.workload, "pipelined": pipelined}))
        return

    subs = {}
    if not args.headline_only:
        for name in ("latent", "highres"):
            if name == args.workload:
                continue
            c = W.VERIFY_CONFIGS[name]
            r = measure_verify(api, name, c["B"], args.mode, args.steps, args.warmup, dev, rank, pg,
                               None, pipelined)
            subs[name] = {
                "workload": workload_name(argparse.Namespace(workload=name, mode=args.mode), c["B"], c["L"],
                                          c["d"], c["dtype"]),
                "value": whole_job_rate(world, c["B"] * c["L"], r["ms_step"] * 1e-3), "unit": UNIT,
                "ms_per_step": r["ms_step"], "steady_state_ms_per_step": r["ms_steady"],
                "hbm_gbs_step": r["roofline"]["algorithmic_bytes"] / (r["ms_step"] * 1e-3) / 1e9,
                "roofline": r["roofline"], "mean_tau_block": r["taus"]["block"],
                "mean_tau_sample": r["taus"]["sample"],
                "gpu_launches": launches_per_step(c["B"], c["d"], pipelined) * args.steps}
        subs["sampler"] = sampler_summary(api, dev)

    e2e_steps = max(20, min(400, args.steps))
    e2e_s, h2d, d2h = measure_e2e(api, head["host0"], Bn, L, d, dt_name, args.mode, dev, e2e_steps)

    nbytes = head["roofline"]["algorithmic_bytes"]
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": head["ms_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32" if dt_name == "f32" else "bf16",
        "data": "synthetic",
        "config": {"workload": workload_name(args, Bn, L, d, dt_name),
                   "global_batch": world * Bn, "window": L, "dim": d,
                   "parallelism": "replicas" if world > 1 else "single-gpu",
                   "l2": "%d rotating input sets, %.0f MB > L2 %.0f MB" % (
                       head["n_sets"], head["n_sets"] * head["set_bytes"] / 1e6, head["l2"] / 1e6)
                   if head["n_sets"] > 1 else "one input set of %.0f MB > L2" % (head["set_bytes"] / 1e6),
                   "cuda_graph": True,
                   "calls": "sdv_verify_pipelined (consecutive independent calls may overlap)"
                            if pipelined else "sdv_verify_ex"},
        "hbm_gbs_step": nbytes / (head["ms_step"] * 1e-3) / 1e9,
        "steady_state": {"ms_per_step": head["ms_steady"], "calls": head["steady_calls"],
                         "value": whole_job_rate(world, Bn * L, head["ms_steady"] * 1e-3),
                         "hbm_gbs": nbytes / (head["ms_steady"] * 1e-3) / 1e9},
        "mean_tau_block": head["taus"]["block"], "mean_tau_sample": head["taus"]["sample"],
        "roofline": head["roofline"],
        "e2e": {"value": world * Bn * L / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h,
                "api": "api.HostStream (pinned [3,B,L,d] window in, accepted_len and y out, "
                       "copy of step i+1 overlapping step i)"},
        "gpu_launches": launches_per_step(Bn, d, pipelined) * args.steps,
        "clocks": head["clocks"],
        "workloads": subs,
    }
    if rank == 0 and world == 1 and not args.skip_cpu:
        rate, nch, tsec = cpu_oracle_rate(head["host0"], 0, args.mode, args.cpu_seconds)
        line["cpu_baseline"] = {"value": rate, "unit": UNIT, "cores": 1, "kind": "oracle",
                                "sample": "%d chains of the %s batch through oracle.verify "
                                          "(numpy fp64, one thread), %.1f s"
                                          % (nch, args.workload, tsec)}
        if Bn == cfg["B"]:
            nproc = max(1, min(os.cpu_count() or 1, Bn))
            prate, pch, pt = cpu_oracle_rate_all_cores(args.workload, Bn, input_seed(cfg["seed"], 0, 0),
                                                       args.mode, args.cpu_seconds, nproc)
            line["cpu_baseline_all_cores"] = {
                "value": prate, "unit": UNIT, "cores": nproc, "kind": "oracle",
                "sample": "%d chains of the %s batch through oracle.verify (numpy fp64) in %d "
                          "spawned processes of one thread, %.1f s each" % (pch, args.workload, nproc, pt)}
    if rank == 0:
        print(json.dumps(line))
    if pg:
        pg.barrier()
        pg.destroy_process_group()


if __name__ == "__main__":
    main()
