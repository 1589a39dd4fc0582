"""Torch-facing helpers over the C ABI: allocate outputs and workspace, pass pointers.

PyTorch provides device memory and the current stream only; every step of the
verification path runs in libspecdiff's kernels.  Inputs must be CUDA tensors
(this module never computes anything itself and has no CPU path).
"""
import torch

from . import binding as B

_DTYPES = {torch.float32: B.SDV_F32, torch.bfloat16: B.SDV_BF16}
_MODES = {"sample": B.SDV_MODE_SAMPLE, "block": B.SDV_MODE_BLOCK,
          B.SDV_MODE_SAMPLE: B.SDV_MODE_SAMPLE, B.SDV_MODE_BLOCK: B.SDV_MODE_BLOCK}
_RESIDUALS = {"decomposition": B.SDV_RESIDUAL_DECOMPOSITION,
              "reflection": B.SDV_RESIDUAL_REFLECTION}


def _ptr(t):
    return 0 if t is None else t.data_ptr()


def _stream():
    return torch.cuda.current_stream().cuda_stream


def _need_cuda(*ts):
    for t in ts:
        if t is not None and (not t.is_cuda or not t.is_contiguous()):
            raise ValueError("libspecdiff needs contiguous CUDA tensors")


def workspace_bytes(B_, L, d, dtype=torch.float32):
    return B.sdv_workspace_bytes(B_, L, d, _DTYPES[dtype])


def make_workspace(B_, L, d, dtype=torch.float32, device="cuda"):
    """A workspace for calls of up to (B_, L, d) (zeroed, though no call needs that)."""
    return torch.zeros(max(workspace_bytes(B_, L, d, dtype), 256), dtype=torch.uint8, device=device)


def _sigma_args(sigma, Bn, L):
    if sigma.dim() == 1:
        if sigma.shape[0] != L:
            raise ValueError("sigma [L] expected")
        return sigma, 0
    if tuple(sigma.shape) != (Bn, L):
        raise ValueError("sigma [B, L] expected")
    return sigma, L


def verify(x_draft, mu_target, mu_draft, sigma, seed, mode="block", *, L_eff=None,
           mu_target_bonus=None, sigma_bonus=None, residual="decomposition", omega=1.0,
           with_ratios=True, with_aux=False, workspace=None, out=None, pipelined=False):
    """One verification call (sdv_verify_ex) on [B, L, d] CUDA tensors; returns a dict of outputs.

    pipelined=True calls sdv_verify_pipelined instead: the call may overlap the end of the
    previous kernel on the stream (see its preconditions in include/specdiff.h)."""
    _need_cuda(x_draft, mu_target, mu_draft, sigma, L_eff, mu_target_bonus, sigma_bonus)
    Bn, L, d = x_draft.shape
    dt = x_draft.dtype
    if mu_target.dtype != dt or mu_draft.dtype != dt or dt not in _DTYPES:
        raise ValueError("x_draft, mu_target, mu_draft must share a float32/bfloat16 dtype")
    if sigma.dtype != torch.float32:
        raise ValueError("sigma must be float32")
    sigma, sstride = _sigma_args(sigma, Bn, L)
    dev = x_draft.device
    if out is None:
        out = {}
    acc = out.get("accepted_len")
    if acc is None:
        acc = torch.empty(Bn, dtype=torch.int32, device=dev)
    y = out.get("y")
    if y is None:
        y = torch.empty(Bn, d, dtype=dt, device=dev)
    lr = dn = None
    if with_ratios:
        lr = out.get("log_ratio")
        lr = torch.empty(Bn, L, dtype=torch.float32, device=dev) if lr is None else lr
        dn = out.get("delta_norm")
        dn = torch.empty(Bn, L, dtype=torch.float32, device=dev) if dn is None else dn
    st = out.get("status")
    st = torch.empty(Bn, dtype=torch.int32, device=dev) if st is None else st
    aux = None
    if with_aux:
        aux = out.get("aux")
        aux = torch.empty(Bn, 4, dtype=torch.float32, device=dev) if aux is None else aux
    if workspace is None:
        workspace = make_workspace(Bn, L, d, dt, dev)
    fn = B.sdv_verify_pipelined if pipelined else B.sdv_verify_ex
    fn(_ptr(x_draft), _ptr(mu_target), _ptr(mu_draft), _ptr(sigma), sstride,
       Bn, L, d, _DTYPES[dt], int(seed) & 0xFFFFFFFFFFFFFFFF, _MODES[mode],
       _ptr(L_eff), _ptr(mu_target_bonus), _ptr(sigma_bonus),
       _RESIDUALS[residual], float(omega),
       _ptr(acc), _ptr(y), _ptr(lr), _ptr(dn), _ptr(st), _ptr(aux),
       _ptr(workspace), workspace.numel(), _stream())
    res = dict(accepted_len=acc, y=y, status=st)
    if with_ratios:
        res.update(log_ratio=lr, delta_norm=dn)
    if with_aux:
        res["aux"] = aux
    return res


def verify_host(x_draft, mu_target, mu_draft, sigma, seed, mode="block", *, dev_bufs=None):
    """End-to-end call from pinned host tensors: copy in, verify, copy accepted_len and y back.

    ``dev_bufs`` (from ``make_device_buffers``) holds the device copies and
    outputs so repeated calls allocate nothing.  Returns (accepted_len, y) as
    host tensors, synchronised.
    """
    Bn, L, d = x_draft.shape
    if dev_bufs is None:
        dev_bufs = make_device_buffers(Bn, L, d, x_draft.dtype, sigma.shape)
    db = dev_bufs
    db["x"].copy_(x_draft, non_blocking=True)
    db["mq"].copy_(mu_target, non_blocking=True)
    db["mp"].copy_(mu_draft, non_blocking=True)
    db["sigma"].copy_(sigma, non_blocking=True)
    verify(db["x"], db["mq"], db["mp"], db["sigma"], seed, mode, with_ratios=False,
           workspace=db["ws"], out=db)
    db["h_acc"].copy_(db["accepted_len"], non_blocking=True)
    db["h_y"].copy_(db["y"], non_blocking=True)
    torch.cuda.current_stream().synchronize()
    return db["h_acc"], db["h_y"]


class HostStream:
    """End-to-end verification of a sequence of windows held in pinned host memory.

    Each window is one pinned host tensor [3, B, L, d] (x_draft, mu_target, mu_draft
    stacked, so that it crosses to the device in one copy) plus sigma.  ``depth`` device
    slots are used in turn: the copy of a window into its slot (on a copy stream)
    overlaps the verification of the previous one (on a compute stream), and each slot's
    accepted lengths and states come back to pinned host memory on the compute stream.
    ``submit`` returns the slot index; ``result`` waits for that slot and returns its
    host tensors (valid until the slot is submitted again).  torch only allocates
    memory and supplies the streams and events; the verification runs in libspecdiff.
    """

    def __init__(self, Bn, L, d, dtype=torch.float32, sigma_shape=None, depth=2, device="cuda"):
        self.Bn, self.L, self.d, self.depth = Bn, L, d, depth
        sigma_shape = (Bn, L) if sigma_shape is None else tuple(sigma_shape)
        self.copy_stream = torch.cuda.Stream(device=device)
        self.compute_stream = torch.cuda.Stream(device=device)
        self.ws = torch.zeros(max(workspace_bytes(Bn, L, d, dtype), 256), dtype=torch.uint8, device=device)
        self.slots = []
        for _ in range(depth):
            self.slots.append(dict(
                win=torch.empty(3, Bn, L, d, dtype=dtype, device=device),
                sigma=torch.empty(*sigma_shape, dtype=torch.float32, device=device),
                accepted_len=torch.empty(Bn, dtype=torch.int32, device=device),
                y=torch.empty(Bn, d, dtype=dtype, device=device),
                status=torch.empty(Bn, dtype=torch.int32, device=device),
                h_acc=torch.empty(Bn, dtype=torch.int32, pin_memory=True),
                h_y=torch.empty(Bn, d, dtype=dtype, pin_memory=True),
                copied=torch.cuda.Event(), done=torch.cuda.Event(), busy=False))
        self.next = 0

    def submit(self, window, sigma, seed, mode="block"):
        i = self.next
        self.next = (i + 1) % self.depth
        sl = self.slots[i]
        if sl["busy"]:
            self.copy_stream.wait_event(sl["done"])      # the slot's previous window is verified
        with torch.cuda.stream(self.copy_stream):
            sl["win"].copy_(window, non_blocking=True)
            sl["sigma"].copy_(sigma, non_blocking=True)
            sl["copied"].record(self.copy_stream)
        self.compute_stream.wait_event(sl["copied"])
        with torch.cuda.stream(self.compute_stream):
            w = sl["win"]
            verify(w[0], w[1], w[2], sl["sigma"], seed, mode, with_ratios=False, workspace=self.ws, out=sl)
            sl["h_acc"].copy_(sl["accepted_len"], non_blocking=True)
            sl["h_y"].copy_(sl["y"], non_blocking=True)
            sl["done"].record(self.compute_stream)
        sl["busy"] = True
        return i

    def result(self, i):
        sl = self.slots[i]
        sl["done"].synchronize()
        return sl["h_acc"], sl["h_y"]


def make_device_buffers(Bn, L, d, dtype, sigma_shape, device="cuda"):
    return dict(
        x=torch.empty(Bn, L, d, dtype=dtype, device=device),
        mq=torch.empty(Bn, L, d, dtype=dtype, device=device),
        mp=torch.empty(Bn, L, d, dtype=dtype, device=device),
        sigma=torch.empty(*sigma_shape, dtype=torch.float32, device=device),
        accepted_len=torch.empty(Bn, dtype=torch.int32, device=device),
        y=torch.empty(Bn, d, dtype=dtype, device=device),
        status=torch.empty(Bn, dtype=torch.int32, device=device),
        ws=make_workspace(Bn, L, d, dtype, device),
        h_acc=torch.empty(Bn, dtype=torch.int32, pin_memory=True),
        h_y=torch.empty(Bn, d, dtype=dtype, pin_memory=True),
    )


def log_ratios(x_draft, mu_target, mu_draft, sigma, L_eff=None, workspace=None):
    """ell_j and |Delta_j| only (sdv_log_ratios)."""
    _need_cuda(x_draft, mu_target, mu_draft, sigma, L_eff)
    Bn, L, d = x_draft.shape
    sigma, sstride = _sigma_args(sigma, Bn, L)
    lr = torch.empty(Bn, L, dtype=torch.float32, device=x_draft.device)
    dn = torch.empty_like(lr)
    if workspace is None:
        workspace = make_workspace(Bn, L, d, x_draft.dtype, x_draft.device)
    B.sdv_log_ratios(_ptr(x_draft), _ptr(mu_target), _ptr(mu_draft), _ptr(sigma), sstride,
                     Bn, L, d, _DTYPES[x_draft.dtype], _ptr(L_eff), _ptr(lr), _ptr(dn),
                     _ptr(workspace), workspace.numel(), _stream())
    return lr, dn


def accept_scan(log_ratio, delta_norm, seed, mode="block", L_eff=None, omega=1.0):
    """tau and log alpha_{tau-1} from given ell, |Delta| (sdv_accept_scan)."""
    _need_cuda(log_ratio, delta_norm, L_eff)
    Bn, L = log_ratio.shape
    tau = torch.empty(Bn, dtype=torch.int32, device=log_ratio.device)
    la = torch.empty(Bn, dtype=torch.float32, device=log_ratio.device)
    B.sdv_accept_scan(_ptr(log_ratio), _ptr(delta_norm), Bn, L, _ptr(L_eff),
                      int(seed) & 0xFFFFFFFFFFFFFFFF, _MODES[mode], float(omega),
                      _ptr(tau), _ptr(la), _stream())
    return tau, la


def usample(delta_norm, log_alpha, w_bits):
    """U = Psi_alpha^{-1}(w) for each item (sdv_usample); w_bits is int32 holding uint32 words."""
    _need_cuda(delta_norm, log_alpha, w_bits)
    n = delta_norm.numel()
    U = torch.empty(n, dtype=torch.float32, device=delta_norm.device)
    st = torch.empty(n, dtype=torch.int32, device=delta_norm.device)
    B.sdv_usample(_ptr(delta_norm), _ptr(log_alpha), _ptr(w_bits), n, _ptr(U), _ptr(st), _stream())
    return U, st


def philox(ctr, seed):
    """Raw Philox4x32-10 blocks for counters ctr [n, 4] (int32 holding uint32 words)."""
    _need_cuda(ctr)
    out = torch.empty_like(ctr)
    B.sdv_philox(_ptr(ctr), int(seed) & 0xFFFFFFFFFFFFFFFF, ctr.shape[0], _ptr(out), _stream())
    return out


def normals(seed, Bn, d, stream_id, sub=0, device="cuda"):
    out = torch.empty(Bn, d, dtype=torch.float32, device=device)
    B.sdv_normals(int(seed) & 0xFFFFFFFFFFFFFFFF, Bn, d, stream_id, sub, _ptr(out), _stream())
    return out


def special(which, z):
    """The device special functions (sdv_special): 'erfcx', 'log_ndtr' or 'gprime' at z (fp32)."""
    _need_cuda(z)
    out = torch.empty_like(z)
    B.sdv_special({"erfcx": 0, "log_ndtr": 1, "gprime": 2}[which], _ptr(z), z.numel(), _ptr(out), _stream())
    return out


class GmmTarget:
    """Analytic Gaussian-mixture target and its variance-preserving schedule (device copies)."""

    def __init__(self, means, log_weights, comp_var, K, churn, beta_min=0.1, beta_max=20.0,
                 t_floor=1e-4, device="cuda"):
        self.means = torch.as_tensor(means, dtype=torch.float32).to(device).contiguous()
        self.log_weights = torch.as_tensor(log_weights, dtype=torch.float32).to(device).contiguous()
        self.C, self.d = self.means.shape
        self.comp_var = float(comp_var)
        self.K = int(K)
        self.churn = float(churn)
        self.beta_min, self.beta_max, self.t_floor = float(beta_min), float(beta_max), float(t_floor)

    def sched(self):
        return (self.K, self.churn, self.beta_min, self.beta_max, self.t_floor)

    def params(self):
        return (_ptr(self.means), _ptr(self.log_weights), self.C, self.comp_var) + self.sched()


def gmm_target(states, k, target):
    """m^q_k(state) and the score for rows of states [n, d] (sdv_gmm_target)."""
    _need_cuda(states, k)
    n, d = states.shape
    mq = torch.empty_like(states)
    sc = torch.empty_like(states)
    B.sdv_gmm_target(_ptr(states), _ptr(k), n, d, *target.params(), _ptr(mq), _ptr(sc), _stream())
    return mq, sc


def free_draft(y, score, k, L_eff, L, target, seed):
    """The drafter's gamma_b steps (sdv_free_draft): x_draft, mu_draft [B, L, d], sigma [B, L]."""
    _need_cuda(y, score, k, L_eff)
    Bn, d = y.shape
    x = torch.zeros(Bn, L, d, dtype=torch.float32, device=y.device)
    mp = torch.zeros_like(x)
    sg = torch.zeros(Bn, L, dtype=torch.float32, device=y.device)
    B.sdv_free_draft(_ptr(y), _ptr(score), _ptr(k), _ptr(L_eff), Bn, L, d, *target.sched(),
                     int(seed) & 0xFFFFFFFFFFFFFFFF, _ptr(x), _ptr(mp), _ptr(sg), _stream())
    return x, mp, sg


def sampler_run(Bn, L, target, seed, mode="block", drafter="free", max_rounds=None,
                workspace=None):
    """Speculative sampling of Bn chains to step K (sdv_sampler_run); returns a dict."""
    dev = target.means.device
    d = target.d
    if workspace is None:
        workspace = torch.empty(B.sdv_sampler_workspace_bytes(Bn, L, d), dtype=torch.uint8,
                                device=dev)
    y = torch.empty(Bn, d, dtype=torch.float32, device=dev)
    k = torch.empty(Bn, dtype=torch.int32, device=dev)
    cr = torch.empty(Bn, dtype=torch.int32, device=dev)
    ts = torch.empty(Bn, dtype=torch.int32, device=dev)
    dr = {"free": B.SDV_DRAFTER_FREE, "frozen": B.SDV_DRAFTER_FROZEN}[drafter]
    mr = target.K if max_rounds is None else int(max_rounds)
    rounds = B.sdv_sampler_run(Bn, L, d, *target.params(), int(seed) & 0xFFFFFFFFFFFFFFFF,
                               _MODES[mode], dr, mr, _ptr(y), _ptr(k), _ptr(cr), _ptr(ts),
                               _ptr(workspace), workspace.numel(), _stream())
    return dict(y=y, k=k, chain_rounds=cr, tau_sum=ts, rounds=rounds)


def sampler_rounds(Bn, L, target, seed, rounds, mode="block", drafter="free", workspace=None):
    """The same sampler driven from the host: sdv_sampler_begin, `rounds` calls of
    sdv_sampler_round, sdv_sampler_end; returns the dict of sampler_run."""
    dev = target.means.device
    d = target.d
    if workspace is None:
        workspace = torch.empty(B.sdv_sampler_workspace_bytes(Bn, L, d), dtype=torch.uint8,
                                device=dev)
    y = torch.empty(Bn, d, dtype=torch.float32, device=dev)
    k = torch.empty(Bn, dtype=torch.int32, device=dev)
    cr = torch.empty(Bn, dtype=torch.int32, device=dev)
    ts = torch.empty(Bn, dtype=torch.int32, device=dev)
    dr = {"free": B.SDV_DRAFTER_FREE, "frozen": B.SDV_DRAFTER_FROZEN}[drafter]
    sd = int(seed) & 0xFFFFFFFFFFFFFFFF
    ws, nb, st = _ptr(workspace), workspace.numel(), _stream()
    B.sdv_sampler_begin(Bn, L, d, *target.params(), sd, ws, nb, st)
    for _ in range(int(rounds)):
        B.sdv_sampler_round(Bn, L, d, *target.params(), sd, _MODES[mode], dr, ws, nb, st)
    r = B.sdv_sampler_end(Bn, L, d, ws, nb, _ptr(y), _ptr(k), _ptr(cr), _ptr(ts), st)
    return dict(y=y, k=k, chain_rounds=cr, tau_sum=ts, rounds=r)


def em_sample(Bn, target, seed):
    """The plain Euler-Maruyama chain (sdv_em_sample)."""
    y = torch.empty(Bn, target.d, dtype=torch.float32, device=target.means.device)
    B.sdv_em_sample(Bn, target.d, *target.params(), int(seed) & 0xFFFFFFFFFFFFFFFF, _ptr(y),
                    _stream())
    return y
