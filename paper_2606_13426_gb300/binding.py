"""ctypes binding of libspecdiff.so: the C-ABI entry points of include/specdiff.h, same names.

Argument marshalling only: every function takes plain integers for device
pointers (0 for NULL) and the cudaStream_t handle, calls the C entry point and
raises ``SDVError`` on a non-zero return code.  The library is loaded on first
use; a missing library raises instead of falling back to anything else.
"""
import ctypes
import os
import threading

from .buildlib import lib_path

SDV_OK = 0
SDV_EINVAL = -1
SDV_EALIGN = -2
SDV_ECUDA = -3
SDV_ENOWORKSPACE = -4

SDV_MODE_SAMPLE = 0
SDV_MODE_BLOCK = 1
SDV_F32 = 0
SDV_BF16 = 1
SDV_RESIDUAL_DECOMPOSITION = 0
SDV_RESIDUAL_REFLECTION = 1
SDV_STATUS_ZERO_DELTA = 1
SDV_STATUS_NONFINITE = 2
SDV_STATUS_USAMPLE_RANGE = 4
SDV_MAX_L = 64
SDV_MAX_COMPONENTS = 16
SDV_DRAFTER_FREE = 0
SDV_DRAFTER_FROZEN = 1
SDV_NOALLOC_SCRATCH_BYTES = 1 << 22

_P = ctypes.c_void_p
_I = ctypes.c_int
_I64 = ctypes.c_int64
_U64 = ctypes.c_uint64
_U32 = ctypes.c_uint32
_F = ctypes.c_float
_SZ = ctypes.c_size_t

# name -> (restype, argtypes); mirrors include/specdiff.h
SIGNATURES = {
    "sdv_version": (ctypes.c_char_p, []),
    "sdv_strerror": (ctypes.c_char_p, [_I]),
    "sdv_last_cuda_error": (_I, []),
    "sdv_workspace_bytes": (_SZ, [_I, _I, _I64, _I]),
    "sdv_verify": (_I, [_P, _P, _P, _P, _I64, _I, _I, _I64, _I, _U64, _I,
                        _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "sdv_verify_ex": (_I, [_P, _P, _P, _P, _I64, _I, _I, _I64, _I, _U64, _I,
                           _P, _P, _P, _I, _F,
                           _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "sdv_verify_pipelined": (_I, [_P, _P, _P, _P, _I64, _I, _I, _I64, _I, _U64, _I,
                                  _P, _P, _P, _I, _F,
                                  _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "sdv_verify_noalloc": (_I, [_P, _P, _P, _P, _I64, _I, _I, _I64, _I, _U64, _I,
                                _P, _P, _P, _P, _P, _P]),
    "sdv_log_ratios": (_I, [_P, _P, _P, _P, _I64, _I, _I, _I64, _I, _P, _P, _P, _P, _SZ, _P]),
    "sdv_accept_scan": (_I, [_P, _P, _I, _I, _P, _U64, _I, _F, _P, _P, _P]),
    "sdv_usample": (_I, [_P, _P, _P, _I, _P, _P, _P]),
    "sdv_philox": (_I, [_P, _U64, _I, _P, _P]),
    "sdv_normals": (_I, [_U64, _I, _I64, _I, _U32, _P, _P]),
    "sdv_special": (_I, [_I, _P, _I, _P, _P]),
    "sdv_gmm_target": (_I, [_P, _P, _I, _I64, _P, _P, _I, _F, _I, _F, _F, _F, _F, _P, _P, _P]),
    "sdv_free_draft": (_I, [_P, _P, _P, _P, _I, _I, _I64, _I, _F, _F, _F, _F, _U64, _P, _P, _P,
                            _P]),
    "sdv_sampler_workspace_bytes": (_SZ, [_I, _I, _I64]),
    "sdv_sampler_run": (_I, [_I, _I, _I64, _P, _P, _I, _F, _I, _F, _F, _F, _F, _U64, _I, _I, _I,
                             _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "sdv_sampler_begin": (_I, [_I, _I, _I64, _P, _P, _I, _F, _I, _F, _F, _F, _F, _U64, _P, _SZ, _P]),
    "sdv_sampler_round": (_I, [_I, _I, _I64, _P, _P, _I, _F, _I, _F, _F, _F, _F, _U64, _I, _I, _P,
                               _SZ, _P]),
    "sdv_sampler_end": (_I, [_I, _I, _I64, _P, _SZ, _P, _P, _P, _P, _P, _P]),
    "sdv_em_sample": (_I, [_I, _I64, _P, _P, _I, _F, _I, _F, _F, _F, _F, _U64, _P, _P]),
    "sdv_timing_enable": (_I, [_I]),
    "sdv_timing_stride": (_I, [_I]),
    "sdv_timing_read": (_I, [_I, _P]),
}

_lib = None
_lock = threading.Lock()


class SDVError(RuntimeError):
    def __init__(self, name, code, cuda_error=0):
        self.code = code
        self.cuda_error = cuda_error
        msg = "%s returned %d (%s)" % (name, code, strerror(code))
        if code == SDV_ECUDA:
            msg += ", cudaError %d" % cuda_error
        super().__init__(msg)


def load(path=None):
    """Load libspecdiff.so (default: the in-tree build) and attach the signatures."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = path or lib_path()
        if not os.path.exists(path):
            raise RuntimeError("libspecdiff.so is not built (%s); run __graft_entry__.build()" % path)
        lib = ctypes.CDLL(path)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def strerror(code):
    if _lib is None:
        return str(code)
    return _lib.sdv_strerror(code).decode()


def _call(name, *args):
    lib = load()
    rc = getattr(lib, name)(*args)
    if rc != SDV_OK:
        raise SDVError(name, rc, lib.sdv_last_cuda_error() if rc == SDV_ECUDA else 0)
    return rc


def sdv_version():
    return load().sdv_version().decode()


def sdv_last_cuda_error():
    return load().sdv_last_cuda_error()


def sdv_workspace_bytes(B, L, d, dtype):
    return int(load().sdv_workspace_bytes(B, L, d, dtype))


def sdv_verify(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed, mode,
               accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
               workspace, workspace_bytes, stream):
    return _call("sdv_verify", x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d,
                 dtype, seed, mode, accepted_len, y_out, log_ratio_out, delta_norm_out,
                 status_out, workspace, workspace_bytes, stream)


def sdv_verify_ex(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                  mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                  accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                  chain_aux_out, workspace, workspace_bytes, stream):
    return _call("sdv_verify_ex", x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d,
                 dtype, seed, mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                 accepted_len, y_out, log_ratio_out, delta_norm_out, status_out, chain_aux_out,
                 workspace, workspace_bytes, stream)


def sdv_verify_pipelined(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                         mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                         accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                         chain_aux_out, workspace, workspace_bytes, stream):
    return _call("sdv_verify_pipelined", x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L,
                 d, dtype, seed, mode, L_eff, mu_target_bonus, sigma_bonus, residual_kind, omega,
                 accepted_len, y_out, log_ratio_out, delta_norm_out, status_out, chain_aux_out,
                 workspace, workspace_bytes, stream)


def sdv_verify_noalloc(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, seed,
                       mode, accepted_len, y_out, log_ratio_out, delta_norm_out, status_out,
                       stream):
    """sdv_verify with its scratch in the library's static device array (no workspace)."""
    return _call("sdv_verify_noalloc", x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L,
                 d, dtype, seed, mode, accepted_len, y_out, log_ratio_out, delta_norm_out,
                 status_out, stream)


def sdv_log_ratios(x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d, dtype, L_eff,
                   log_ratio_out, delta_norm_out, workspace, workspace_bytes, stream):
    return _call("sdv_log_ratios", x_draft, mu_target, mu_draft, sigma, sigma_stride_b, B, L, d,
                 dtype, L_eff, log_ratio_out, delta_norm_out, workspace, workspace_bytes, stream)


def sdv_accept_scan(log_ratio, delta_norm, B, L, L_eff, seed, mode, omega, tau_out,
                    log_alpha_res_out, stream):
    return _call("sdv_accept_scan", log_ratio, delta_norm, B, L, L_eff, seed, mode, omega,
                 tau_out, log_alpha_res_out, stream)


def sdv_usample(delta_norm, log_alpha, w_bits, n, U_out, status_out, stream):
    return _call("sdv_usample", delta_norm, log_alpha, w_bits, n, U_out, status_out, stream)


def sdv_philox(ctr, seed, n, out, stream):
    return _call("sdv_philox", ctr, seed, n, out, stream)


def sdv_normals(seed, B, d, stream_id, sub, out, stream):
    return _call("sdv_normals", seed, B, d, stream_id, sub, out, stream)


def sdv_special(which, z, n, out, stream):
    return _call("sdv_special", which, z, n, out, stream)


def sdv_timing_enable(slots):
    return _call("sdv_timing_enable", slots)


def sdv_timing_stride(every):
    return _call("sdv_timing_stride", every)


def sdv_timing_read(n_calls):
    """Summed (K1, K2, K4) milliseconds of the last n_calls recorded calls."""
    ms = (ctypes.c_float * 3)()
    _call("sdv_timing_read", n_calls, ctypes.addressof(ms))
    return [float(v) for v in ms]


def sdv_gmm_target(states, k, n, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max,
                   t_floor, mq_out, score_out, stream):
    return _call("sdv_gmm_target", states, k, n, d, means, log_weights, C, comp_var, K, churn,
                 beta_min, beta_max, t_floor, mq_out, score_out, stream)


def sdv_free_draft(y, score, k, L_eff, B, L, d, K, churn, beta_min, beta_max, t_floor, seed,
                   x_draft, mu_draft, sigma, stream):
    return _call("sdv_free_draft", y, score, k, L_eff, B, L, d, K, churn, beta_min, beta_max,
                 t_floor, seed, x_draft, mu_draft, sigma, stream)


def sdv_sampler_workspace_bytes(B, L, d):
    return int(load().sdv_sampler_workspace_bytes(B, L, d))


def sdv_sampler_run(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max,
                    t_floor, seed, mode, drafter, max_rounds, y_out, k_out, chain_rounds_out,
                    tau_sum_out, workspace, workspace_bytes, stream):
    """Returns the number of rounds run (the C call's rounds_out)."""
    rounds = ctypes.c_int32(0)
    _call("sdv_sampler_run", B, L, d, means, log_weights, C, comp_var, K, churn, beta_min,
          beta_max, t_floor, seed, mode, drafter, max_rounds, y_out, k_out, chain_rounds_out,
          tau_sum_out, ctypes.addressof(rounds), workspace, workspace_bytes, stream)
    return int(rounds.value)


def sdv_sampler_begin(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max,
                      t_floor, seed, workspace, workspace_bytes, stream):
    return _call("sdv_sampler_begin", B, L, d, means, log_weights, C, comp_var, K, churn, beta_min,
                 beta_max, t_floor, seed, workspace, workspace_bytes, stream)


def sdv_sampler_round(B, L, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max,
                      t_floor, seed, mode, drafter, workspace, workspace_bytes, stream):
    return _call("sdv_sampler_round", B, L, d, means, log_weights, C, comp_var, K, churn, beta_min,
                 beta_max, t_floor, seed, mode, drafter, workspace, workspace_bytes, stream)


def sdv_sampler_end(B, L, d, workspace, workspace_bytes, y_out, k_out, chain_rounds_out,
                    tau_sum_out, stream):
    """Returns the number of rounds run (the C call's rounds_out)."""
    rounds = ctypes.c_int32(0)
    _call("sdv_sampler_end", B, L, d, workspace, workspace_bytes, y_out, k_out, chain_rounds_out,
          tau_sum_out, ctypes.addressof(rounds), stream)
    return int(rounds.value)


def sdv_em_sample(B, d, means, log_weights, C, comp_var, K, churn, beta_min, beta_max, t_floor,
                  seed, y_out, stream):
    return _call("sdv_em_sample", B, d, means, log_weights, C, comp_var, K, churn, beta_min,
                 beta_max, t_floor, seed, y_out, stream)
