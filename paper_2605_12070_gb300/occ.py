"""Thin ctypes binding of the occ C ABI (include/occ.h) for torch tensors.

Argument marshalling only: every step of the computation runs in the CUDA
kernels of ``libocc.so``.  The functions carry the C names.  Tensors must be
CUDA tensors; outputs not supplied by the caller are allocated with
``torch.empty`` on the input's device.  Calls are asynchronous on the current
torch stream unless ``stream`` (a ``torch.cuda.Stream``) is given.

There is no CPU fallback: if the library is missing or a tensor is not on a
CUDA device, the call raises.
"""

import contextlib
import ctypes
import math
import os
import struct
import weakref
from dataclasses import dataclass

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libocc.so")

OCC_OK = 0
OCC_F32, OCC_BF16 = 0, 1
FLAG_IN_BAND, FLAG_CLIPPED, FLAG_ACTIVE, FLAG_VALID = 1, 2, 4, 8
DATA_ERR_BAD_ID = 1

LOSS_STATS_BYTES = 64     # sizeof(occ_loss_stats)
EWMA_STATE_BYTES = 40     # sizeof(occ_ewma_state)
_STATS_FMT = "<2d5q2i"
_STATE_FMT = "<3d4i"

# Every symbol declared in include/occ.h.
EXPORTS = ("occ_token_logprob", "occ_loss_workspace_bytes", "occ_decoupled_loss_fwd_bwd",
           "occ_decoupled_loss_fused", "occ_decoupled_loss_fwd_bwd_noalloc", "occ_ewma_update",
           "occ_ewma_update_bf16", "occ_ewma_update_host", "occ_ewma_state_init",
           "occ_host_alloc", "occ_host_free", "occ_status_string", "occ_last_error",
           "occ_last_kernel", "occ_version", "occ_set_option", "occ_get_option")

# occ_option codes (include/occ.h)
OPTIONS = {"k1_warp": 0, "k1_threads": 1, "k2_threads": 2, "k2_head_bytes": 3, "k2_unroll": 4,
           "fused_threads": 5, "fused_head_bytes": 6, "fused_tmem": 7,
           "k2_tmem": 8}


class OccError(RuntimeError):
    pass


class LossParams(ctypes.Structure):
    """Mirror of occ_loss_params (host struct)."""
    _fields_ = [("rd_lo", ctypes.c_double), ("rd_hi", ctypes.c_double),
                ("eps_low", ctypes.c_double), ("eps_high", ctypes.c_double),
                ("grad_scale", ctypes.c_double), ("denom", ctypes.c_int64),
                ("rd_weight", ctypes.c_int32), ("dlogits_f32", ctypes.c_int32),
                ("proxy", ctypes.c_int32), ("reserved", ctypes.c_int32),
                ("alpha", ctypes.c_double)]


PROXY_NONE, PROXY_LOGLINEAR, PROXY_ARITHMETIC = 0, 1, 2
_PROXIES = {None: 0, "none": 0, "loglinear": 1, "arithmetic": 2}


def _params(rd_lo, rd_hi, eps_low, eps_high, grad_scale, denom, rd_weight, dlogits_f32,
            proxy=None, alpha=0.0):
    return LossParams(float(rd_lo), float(rd_hi), float(eps_low), float(eps_high),
                      float(grad_scale), int(denom), int(rd_weight), int(bool(dlogits_f32)),
                      _PROXIES[proxy], 0, float(alpha))


_lib = None


def lib():
    """Loads libocc.so once; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise OccError(f"{LIB_PATH} is not built; run `python -m paper_2605_12070_gb300.build` "
                       "or __graft_entry__.build()")
    L = ctypes.CDLL(LIB_PATH)
    vp, i64, i32, dbl = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_double
    L.occ_token_logprob.argtypes = [vp, i32, i64, i64, i64, vp, vp, vp, vp]
    L.occ_token_logprob.restype = i32
    L.occ_loss_workspace_bytes.argtypes = [i64, i64]
    L.occ_loss_workspace_bytes.restype = ctypes.c_size_t
    L.occ_decoupled_loss_fwd_bwd.argtypes = [vp, i32, i64, i64, i64, vp, vp, vp, vp, vp,
                                             ctypes.POINTER(LossParams), vp, vp, vp, i64, vp, vp,
                                             ctypes.c_size_t, vp]
    L.occ_decoupled_loss_fwd_bwd.restype = i32
    L.occ_decoupled_loss_fused.argtypes = [vp, vp, i32, i64, i64, i64, i64, vp, vp, vp, vp,
                                           ctypes.POINTER(LossParams), vp, vp, vp, vp, vp, vp, i64,
                                           vp, vp, ctypes.c_size_t, vp]
    L.occ_decoupled_loss_fused.restype = i32
    L.occ_decoupled_loss_fwd_bwd_noalloc.argtypes = [vp, i32, i64, i64, i64, vp, vp, vp, vp, vp,
                                                     ctypes.POINTER(LossParams), vp, vp, vp, i64,
                                                     vp, vp]
    L.occ_decoupled_loss_fwd_bwd_noalloc.restype = i32
    L.occ_ewma_update.argtypes = [vp, vp, i64, dbl, vp, vp, dbl, i32, i32, vp]
    L.occ_ewma_update.restype = i32
    u64 = ctypes.c_uint64
    L.occ_ewma_update_bf16.argtypes = [vp, vp, i32, i64, dbl, vp, vp, dbl, i32, i32, u64, vp]
    L.occ_ewma_update_bf16.restype = i32
    L.occ_ewma_update_host.argtypes = [vp, i32, vp, i32, i64, dbl, vp, vp, dbl, i32, i32, u64, vp,
                                       ctypes.c_size_t, vp, vp]
    L.occ_ewma_update_host.restype = i32
    L.occ_ewma_state_init.argtypes = [vp, dbl, vp]
    L.occ_ewma_state_init.restype = i32
    L.occ_host_alloc.argtypes = [ctypes.c_size_t, ctypes.POINTER(vp)]
    L.occ_host_alloc.restype = i32
    L.occ_host_free.argtypes = [vp, ctypes.c_size_t]
    L.occ_host_free.restype = i32
    L.occ_status_string.argtypes = [i32]
    L.occ_status_string.restype = ctypes.c_char_p
    L.occ_last_error.argtypes = []
    L.occ_last_error.restype = ctypes.c_char_p
    L.occ_last_kernel.argtypes = []
    L.occ_last_kernel.restype = ctypes.c_char_p
    L.occ_version.argtypes = []
    L.occ_version.restype = ctypes.c_int
    L.occ_set_option.argtypes = [i32, i64]
    L.occ_set_option.restype = i32
    L.occ_get_option.argtypes = [i32]
    L.occ_get_option.restype = i64
    _lib = L
    return L


def set_option(name, value):
    """Sets a process-wide launch-shape option (-1 = automatic)."""
    _check(lib().occ_set_option(OPTIONS[name], int(value)), f"occ_set_option({name})")


def get_option(name):
    return int(lib().occ_get_option(OPTIONS[name]))


@contextlib.contextmanager
def options(**kw):
    """Sets options for the duration of a block, then restores them."""
    old = {k: get_option(k) for k in kw}
    try:
        for k, v in kw.items():
            set_option(k, v)
        yield
    finally:
        for k, v in old.items():
            set_option(k, v)


def occ_last_kernel():
    """The row kernel that the last occ call on this thread launched ("" if none)."""
    return lib().occ_last_kernel().decode()


def _check(rc, what):
    if rc != OCC_OK:
        L = lib()
        raise OccError(f"{what}: {L.occ_status_string(rc).decode()} "
                       f"({L.occ_last_error().decode()})")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream, device):
    s = stream if stream is not None else torch.cuda.current_stream(device)
    return ctypes.c_void_p(s.cuda_stream)


def _on(device):
    """Makes `device` current for the call: the library launches on the
    current device, which must hold every pointer and the stream."""
    return torch.cuda.device(device)


def _cuda(*ts):
    for t in ts:
        if t is not None and not t.is_cuda:
            raise OccError("occ kernels need CUDA tensors (no CPU fallback)")


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return OCC_BF16
    if t.dtype == torch.float32:
        return OCC_F32
    raise OccError(f"unsupported logits dtype {t.dtype}")


def _rows(logits):
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise OccError("logits must be a 2-D tensor with unit column stride")
    return logits.shape[0], logits.shape[1], logits.stride(0)


def occ_token_logprob(logits, ids, logp_out=None, lse_out=None, want_lse=False, stream=None):
    """log pi(y_t) (and optionally lse) for each row of ``logits`` [T, V]."""
    _cuda(logits, ids, logp_out, lse_out)
    T, V, ld = _rows(logits)
    if logp_out is None:
        logp_out = torch.empty(T, dtype=torch.float32, device=logits.device)
    if lse_out is None and want_lse:
        lse_out = torch.empty(T, dtype=torch.float32, device=logits.device)
    with _on(logits.device):
        rc = lib().occ_token_logprob(_ptr(logits), _dtype_code(logits), T, V, ld, _ptr(ids),
                                     _ptr(logp_out), _ptr(lse_out), _stream(stream, logits.device))
    _check(rc, "occ_token_logprob")
    return logp_out, lse_out


def occ_loss_workspace_bytes(T, V):
    return int(lib().occ_loss_workspace_bytes(int(T), int(V)))


def new_loss_stats(device):
    return torch.zeros(LOSS_STATS_BYTES, dtype=torch.uint8, device=device)


def new_workspace(T, V, device):
    return torch.empty(occ_loss_workspace_bytes(T, V), dtype=torch.uint8, device=device)


@dataclass
class LossStats:
    loss_sum: float
    loss: float
    n_valid: int
    n_rd_out: int
    n_clipped: int
    n_active: int
    denom: int
    err: int

    @property
    def rho(self):
        """Train-Infer Mask value of Sec. 5.2: fraction of valid tokens kept active."""
        return self.n_active / self.n_valid if self.n_valid else float("nan")


def decode_loss_stats(t):
    v = struct.unpack(_STATS_FMT, bytes(t.detach().to("cpu").numpy().tobytes()))
    return LossStats(*v[:8])


def occ_decoupled_loss_fwd_bwd(logits, ids, logp_old, logp_mu, adv, loss_mask=None, *,
                               rd_lo, rd_hi, eps_low, eps_high, rd_weight=1, grad_scale=1.0,
                               denom=0, dlogits_f32=False, dlogits="new", logp_out=None,
                               flags_out=None, want_logp=True, want_flags=True, stats=None,
                               workspace=None, stream=None, proxy=None, alpha=0.0):
    """The decoupled PPO loss over ``logits`` [T, V] and its gradient.

    ``dlogits``: "new" (allocate), None (forward only), "inplace" (overwrite
    ``logits``), or a tensor [T, >=V].  ``proxy`` ("loglinear" or "arithmetic",
    with weight ``alpha``) builds log pi_old per token instead of reading
    ``logp_old`` (which may then be None).  Returns a dict with 'stats' (raw
    device bytes), 'dlogits', 'logp', 'flags'.
    """
    _cuda(logits, ids, logp_old, logp_mu, adv, loss_mask)
    T, V, ld = _rows(logits)
    dev = logits.device
    out_dtype = torch.float32 if (dlogits_f32 or logits.dtype == torch.float32) else logits.dtype
    if isinstance(dlogits, str):
        if dlogits == "new":
            dlogits = torch.empty((T, V), dtype=out_dtype, device=dev)
        elif dlogits == "inplace":
            dlogits = logits
        else:
            raise OccError(f"dlogits={dlogits!r}")
    if dlogits is not None:
        _cuda(dlogits)
        if dlogits.dim() != 2 or dlogits.stride(1) != 1 or dlogits.dtype != out_dtype:
            raise OccError("dlogits must be 2-D, unit column stride, dtype " + str(out_dtype))
    ld_grad = dlogits.stride(0) if dlogits is not None else 0
    if logp_out is None and want_logp:
        logp_out = torch.empty(T, dtype=torch.float32, device=dev)
    if flags_out is None and want_flags:
        flags_out = torch.empty(T, dtype=torch.uint8, device=dev)
    if stats is None:
        stats = new_loss_stats(dev)
    if workspace is None:
        workspace = new_workspace(T, V, dev)
    p = _params(rd_lo, rd_hi, eps_low, eps_high, grad_scale, denom, rd_weight, dlogits_f32,
                proxy, alpha)
    with _on(dev):
        rc = lib().occ_decoupled_loss_fwd_bwd(
            _ptr(logits), _dtype_code(logits), T, V, ld, _ptr(ids), _ptr(logp_old), _ptr(logp_mu),
            _ptr(adv), _ptr(loss_mask), ctypes.byref(p), _ptr(logp_out), _ptr(flags_out),
            _ptr(dlogits), ld_grad, _ptr(stats), _ptr(workspace), workspace.numel(),
            _stream(stream, dev))
    _check(rc, "occ_decoupled_loss_fwd_bwd")
    return {"stats": stats, "dlogits": dlogits, "logp": logp_out, "flags": flags_out}


def occ_decoupled_loss_fused(logits, logits_old, ids, logp_mu, adv, loss_mask=None, *, rd_lo,
                             rd_hi, eps_low, eps_high, rd_weight=1, grad_scale=1.0, denom=0,
                             dlogits_f32=False, dlogits="new", logp_out=None, logp_old_out=None,
                             flags_out=None, entropy_out=None, kl_out=None, want_logp=True,
                             want_logp_old=True, want_flags=True, want_diagnostics=False,
                             stats=None, workspace=None, stream=None):
    """log pi_old and the decoupled loss (+ dlogits) in one launch; optional
    per-token entropy of pi_theta and KL(pi_old || pi_theta)."""
    _cuda(logits, logits_old, ids, logp_mu, adv, loss_mask)
    T, V, ld = _rows(logits)
    To, Vo, ld_old = _rows(logits_old)
    if (To, Vo) != (T, V) or logits_old.dtype != logits.dtype:
        raise OccError("logits_old must match logits in shape and dtype")
    dev = logits.device
    out_dtype = torch.float32 if (dlogits_f32 or logits.dtype == torch.float32) else logits.dtype
    if isinstance(dlogits, str):
        if dlogits == "new":
            dlogits = torch.empty((T, V), dtype=out_dtype, device=dev)
        elif dlogits == "inplace":
            dlogits = logits
        else:
            raise OccError(f"dlogits={dlogits!r}")
    if dlogits is not None:
        _cuda(dlogits)
        if dlogits.dim() != 2 or dlogits.stride(1) != 1 or dlogits.dtype != out_dtype:
            raise OccError("dlogits must be 2-D, unit column stride, dtype " + str(out_dtype))
    ld_grad = dlogits.stride(0) if dlogits is not None else 0

    def _f32(t, want):
        return torch.empty(T, dtype=torch.float32, device=dev) if (t is None and want) else t

    logp_out = _f32(logp_out, want_logp)
    logp_old_out = _f32(logp_old_out, want_logp_old)
    entropy_out = _f32(entropy_out, want_diagnostics)
    kl_out = _f32(kl_out, want_diagnostics)
    if flags_out is None and want_flags:
        flags_out = torch.empty(T, dtype=torch.uint8, device=dev)
    if stats is None:
        stats = new_loss_stats(dev)
    if workspace is None:
        workspace = new_workspace(T, V, dev)
    p = _params(rd_lo, rd_hi, eps_low, eps_high, grad_scale, denom, rd_weight, dlogits_f32)
    with _on(dev):
        rc = lib().occ_decoupled_loss_fused(
            _ptr(logits), _ptr(logits_old), _dtype_code(logits), T, V, ld, ld_old, _ptr(ids),
            _ptr(logp_mu), _ptr(adv), _ptr(loss_mask), ctypes.byref(p), _ptr(logp_out),
            _ptr(logp_old_out), _ptr(flags_out), _ptr(entropy_out), _ptr(kl_out), _ptr(dlogits),
            ld_grad, _ptr(stats), _ptr(workspace), workspace.numel(), _stream(stream, dev))
    _check(rc, "occ_decoupled_loss_fused")
    return {"stats": stats, "dlogits": dlogits, "logp": logp_out, "logp_old": logp_old_out,
            "flags": flags_out, "entropy": entropy_out, "kl": kl_out}


NOALLOC_MAX_TOKENS = 786432  # OCC_NOALLOC_MAX_TOKENS


def occ_decoupled_loss_fwd_bwd_noalloc(logits, ids, logp_old, logp_mu, adv, loss_mask, *,
                                       rd_lo, rd_hi, eps_low, eps_high, rd_weight=1,
                                       grad_scale=1.0, denom=0, dlogits_f32=False, dlogits,
                                       logp_out, flags_out, stats, stream=None):
    """occ_decoupled_loss_fwd_bwd for callers that cannot allocate device memory.

    Every output buffer must be supplied (``dlogits`` may be None for a
    forward-only call); the scratch comes from the library's own fixed array,
    so at most NOALLOC_MAX_TOKENS tokens per call, and calls must not overlap
    on the GPU.
    """
    _cuda(logits, ids, logp_old, logp_mu, adv, loss_mask, dlogits, logp_out, flags_out, stats)
    T, V, ld = _rows(logits)
    ld_grad = dlogits.stride(0) if dlogits is not None else 0
    p = _params(rd_lo, rd_hi, eps_low, eps_high, grad_scale, denom, rd_weight, dlogits_f32)
    with _on(logits.device):
        rc = lib().occ_decoupled_loss_fwd_bwd_noalloc(
            _ptr(logits), _dtype_code(logits), T, V, ld, _ptr(ids), _ptr(logp_old), _ptr(logp_mu),
            _ptr(adv), _ptr(loss_mask), ctypes.byref(p), _ptr(logp_out), _ptr(flags_out),
            _ptr(dlogits), ld_grad, _ptr(stats), _stream(stream, logits.device))
    _check(rc, "occ_decoupled_loss_fwd_bwd_noalloc")
    return {"stats": stats, "dlogits": dlogits, "logp": logp_out, "flags": flags_out}


def new_ewma_state(device, w0=0.0, stream=None):
    st = torch.zeros(EWMA_STATE_BYTES, dtype=torch.uint8, device=device)
    occ_ewma_state_init(st, w0, stream)
    return st


def occ_ewma_state_init(state, w0, stream=None):
    _cuda(state)
    with _on(state.device):
        rc = lib().occ_ewma_state_init(_ptr(state), float(w0), _stream(stream, state.device))
    _check(rc, "occ_ewma_state_init")


@dataclass
class EwmaState:
    w: float
    coef_a: float
    coef_b: float
    streak: int
    n_resets: int
    last_reset: int


def decode_ewma_state(t):
    v = struct.unpack(_STATE_FMT, bytes(t.detach().to("cpu").numpy().tobytes()))
    return EwmaState(*v[:6])


def occ_ewma_update(theta_prox, theta, beta, state, stats=None, tau=0.9, min_streak=1,
                    force_reset=False, stream=None):
    """theta_prox <- revised PPO-EWMA step toward theta (in place)."""
    _cuda(theta_prox, theta, state, stats)
    if theta_prox.dtype != torch.float32 or theta.dtype != torch.float32:
        raise OccError("EWMA buffers must be float32")
    if not (theta_prox.is_contiguous() and theta.is_contiguous()):
        raise OccError("EWMA buffers must be contiguous")
    n = theta_prox.numel()
    if theta.numel() != n:
        raise OccError("theta_prox and theta differ in size")
    with _on(theta_prox.device):
        rc = lib().occ_ewma_update(_ptr(theta_prox), _ptr(theta), n, float(beta), _ptr(state),
                                   _ptr(stats), float(tau), int(min_streak), int(bool(force_reset)),
                                   _stream(stream, theta_prox.device))
    _check(rc, "occ_ewma_update")
    return theta_prox


def _float_code(t):
    if t.dtype == torch.bfloat16:
        return OCC_BF16
    if t.dtype == torch.float32:
        return OCC_F32
    raise OccError(f"unsupported dtype {t.dtype}")


def occ_ewma_update_bf16(theta_prox, theta, beta, state, stats=None, tau=0.9, min_streak=1,
                         force_reset=False, sr_seed=0, stream=None):
    """PPO-EWMA step on a bf16 proximal buffer (theta float32 or bf16); sr_seed != 0
    selects stochastic rounding."""
    _cuda(theta_prox, theta, state, stats)
    if theta_prox.dtype != torch.bfloat16 or not theta_prox.is_contiguous() or \
            not theta.is_contiguous() or theta.numel() != theta_prox.numel():
        raise OccError("theta_prox must be contiguous bf16 and match theta")
    with _on(theta_prox.device):
        rc = lib().occ_ewma_update_bf16(_ptr(theta_prox), _ptr(theta), _float_code(theta),
                                        theta_prox.numel(), float(beta), _ptr(state), _ptr(stats),
                                        float(tau), int(min_streak), int(bool(force_reset)),
                                        int(sr_seed), _stream(stream, theta_prox.device))
    _check(rc, "occ_ewma_update_bf16")
    return theta_prox


def occ_ewma_update_host(theta_prox_host, theta, beta, state, staging, stats=None, tau=0.9,
                         min_streak=1, force_reset=False, sr_seed=0, stream0=None, stream1=None):
    """PPO-EWMA step on a pinned host proximal buffer, streamed through ``staging``
    (a device uint8 tensor) on two streams."""
    _cuda(theta, state, stats, staging)
    if theta_prox_host.is_cuda or not theta_prox_host.is_pinned():
        raise OccError("theta_prox_host must be a pinned host tensor")
    dev = theta.device
    s0 = stream0 if stream0 is not None else torch.cuda.current_stream(dev)
    s1 = stream1 if stream1 is not None else s0
    with _on(dev):
        rc = lib().occ_ewma_update_host(
            _ptr(theta_prox_host), _float_code(theta_prox_host), _ptr(theta), _float_code(theta),
            theta.numel(), float(beta), _ptr(state), _ptr(stats), float(tau), int(min_streak),
            int(bool(force_reset)), int(sr_seed), _ptr(staging), staging.numel(),
            ctypes.c_void_p(s0.cuda_stream), ctypes.c_void_p(s1.cuda_stream))
    _check(rc, "occ_ewma_update_host")
    return theta_prox_host


def _host_free(ptr, nbytes):
    lib().occ_host_free(ctypes.c_void_p(ptr), nbytes)


def occ_host_alloc(shape, dtype):
    """Pinned host tensor from occ_host_alloc (huge-page backed, zero-filled).

    The memory is released through occ_host_free when the last tensor or view
    of it is gone; copies from or to it must have completed by then."""
    if isinstance(shape, int):
        shape = (shape,)
    elem = torch.empty((), dtype=dtype).element_size()
    nbytes = math.prod(shape) * elem
    if nbytes == 0:
        return torch.empty(shape, dtype=dtype, pin_memory=True)
    # torch reports a registered range as pinned (and copies it asynchronously)
    # only once its own CUDA state exists
    torch.cuda.init()
    ptr = ctypes.c_void_p()
    _check(lib().occ_host_alloc(nbytes, ctypes.byref(ptr)), "occ_host_alloc")
    buf = (ctypes.c_uint8 * nbytes).from_address(ptr.value)
    weakref.finalize(buf, _host_free, ptr.value, nbytes)
    return torch.frombuffer(buf, dtype=torch.uint8).view(dtype).view(shape)
