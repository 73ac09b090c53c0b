"""Thin ctypes binding of libsolo_readout (argument marshalling only).

Function names match the C ABI in ``include/solo_readout.h``.  Tensors are
PyTorch tensors used for device memory and streams: their data pointers and
the current CUDA stream are handed to the library; every step of the
computation runs in the library's kernels.  There is no fallback: when the
library is missing or the device is not sm_103a the calls raise.
"""
from __future__ import annotations

import ctypes
import os
from typing import Sequence

from . import build as _build

SOLO_OK = 0
SOLO_ERR_INVALID_ARG = -1
SOLO_ERR_UNSUPPORTED_SHAPE = -2
SOLO_ERR_WORKSPACE_TOO_SMALL = -3
SOLO_ERR_CUDA = -4
SOLO_ERR_NOT_SM103 = -5
SOLO_ERR_MISALIGNED = -6
SOLO_ERR_EXCEEDS_STATIC_SCRATCH = -7
SOLO_STATIC_SCRATCH_BYTES = 64 << 20

SOLO_FLAG_BAD_TARGET = 1
SOLO_FLAG_TIMEOUT = 2

SOLO_NUM_STAGES = 8
SOLO_EXIT_NUM_STAGES = 3
SOLO_ONCHIP_NUM_STAGES = 4
ONCHIP_STAGE_NAMES = ["final", "aux_prep", "aux_onchip", "aux_means"]
EXIT_STAGE_NAMES = ["rmsnorm", "logits", "combine"]
STAGE_NAMES = ["rmsnorm", "logits", "lse", "grad", "dxhat", "norm_bwd", "dW", "dgamma"]


class solo_dims_t(ctypes.Structure):
    _fields_ = [("K", ctypes.c_int32), ("N", ctypes.c_int64), ("d", ctypes.c_int32),
                ("V", ctypes.c_int32), ("eps", ctypes.c_float),
                ("ignore_index", ctypes.c_int32)]


class solo_heads_t(ctypes.Structure):
    _fields_ = [("tau", ctypes.c_void_p), ("bias", ctypes.c_void_p), ("dtau", ctypes.c_void_p),
                ("dbias", ctypes.c_void_p)]


class SoloError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {strerror(status)} (status {status})")
        self.status = status


_lib = None


def library_path() -> str:
    """The in-tree release library, or the file named by SOLO_READOUT_LIB (e.g.
    the checked build)."""
    return os.environ.get("SOLO_READOUT_LIB") or _build.LIB


def load(path: str | None = None) -> ctypes.CDLL:
    """Loads the in-tree library (raises when it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or library_path()
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with "
                          "`python -m paper_2609_35440_gb300.build` (needs nvcc)")
    lib = ctypes.CDLL(path)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    dims_p = ctypes.POINTER(solo_dims_t)
    lib.solo_readout_workspace_bytes.argtypes = [dims_p, ctypes.POINTER(sz)]
    lib.solo_readout_workspace_bytes.restype = i32
    common = [dims_p, ctypes.POINTER(vp), vp, vp, vp, vp, vp, vp, ctypes.POINTER(vp), vp, vp,
              vp, sz, vp]
    lib.solo_readout_fwd_bwd.argtypes = common
    lib.solo_readout_fwd_bwd.restype = i32
    lib.solo_readout_fwd_bwd_events.argtypes = common + [ctypes.POINTER(vp), i32]
    lib.solo_readout_fwd_bwd_events.restype = i32
    lib.solo_readout_get_flags.argtypes = [vp, vp, ctypes.POINTER(ctypes.c_uint32)]
    lib.solo_readout_get_flags.restype = i32
    lib.solo_readout_strerror.argtypes = [i32]
    lib.solo_readout_strerror.restype = ctypes.c_char_p
    lib.solo_readout_fwd_bwd_static.argtypes = [dims_p, ctypes.POINTER(vp), vp, vp, vp, vp, vp,
                                                 vp, ctypes.POINTER(vp), vp, vp, vp, vp]
    lib.solo_readout_fwd_bwd_static.restype = i32
    lib.solo_readout_selftest_wait_timeout.argtypes = [vp, ctypes.c_uint32, vp]
    lib.solo_readout_selftest_wait_timeout.restype = i32
    lib.solo_readout_exit_workspace_bytes.argtypes = [dims_p, ctypes.POINTER(sz)]
    lib.solo_readout_exit_workspace_bytes.restype = i32
    lib.solo_readout_exit_forward.argtypes = [dims_p, ctypes.POINTER(vp), vp, vp, vp, vp, vp, vp,
                                              vp, vp, vp, sz, vp]
    lib.solo_readout_exit_forward.restype = i32
    lib.solo_readout_exit_forward_events.argtypes = (
        lib.solo_readout_exit_forward.argtypes + [ctypes.POINTER(vp), i32])
    lib.solo_readout_exit_forward_events.restype = i32
    lib.solo_readout_fwd_bwd_heads.argtypes = [dims_p, ctypes.POINTER(vp), vp, vp, vp, vp,
                                                ctypes.POINTER(solo_heads_t), vp, vp,
                                                ctypes.POINTER(vp), vp, vp, vp, sz, vp,
                                                ctypes.POINTER(vp), i32]
    lib.solo_readout_fwd_bwd_heads.restype = i32
    lib.solo_readout_private_workspace_bytes.argtypes = [dims_p, ctypes.POINTER(sz)]
    lib.solo_readout_private_workspace_bytes.restype = i32
    lib.solo_readout_fwd_bwd_private.argtypes = [dims_p, ctypes.POINTER(vp), ctypes.POINTER(vp),
                                                  ctypes.POINTER(vp), vp, vp,
                                                  ctypes.POINTER(solo_heads_t), vp, vp,
                                                  ctypes.POINTER(vp), ctypes.POINTER(vp),
                                                  ctypes.POINTER(vp), vp, sz, vp]
    lib.solo_readout_fwd_bwd_private.restype = i32
    lib.solo_readout_version.argtypes = []
    lib.solo_readout_version.restype = i32
    lib.solo_readout_kernel_launches.argtypes = []
    lib.solo_readout_kernel_launches.restype = ctypes.c_uint64
    lib.solo_readout_build_flags.argtypes = []
    lib.solo_readout_build_flags.restype = i32
    lib.solo_readout_rmsnorm.argtypes = [dims_p, ctypes.POINTER(vp), vp, vp, vp, vp]
    lib.solo_readout_rmsnorm.restype = i32
    lib.solo_readout_onchip_workspace_bytes.argtypes = [dims_p, ctypes.POINTER(sz)]
    lib.solo_readout_onchip_workspace_bytes.restype = i32
    lib.solo_readout_fwd_bwd_onchip.argtypes = common + [ctypes.POINTER(vp), i32]
    lib.solo_readout_fwd_bwd_onchip.restype = i32
    _lib = lib
    return lib


def strerror(status: int) -> str:
    return load().solo_readout_strerror(int(status)).decode()


def make_dims(K: int, N: int, d: int, V: int, eps: float = 1e-6,
              ignore_index: int = -100) -> solo_dims_t:
    return solo_dims_t(K, N, d, V, eps, ignore_index)


def solo_readout_workspace_bytes(dims: solo_dims_t) -> int:
    out = ctypes.c_size_t(0)
    st = load().solo_readout_workspace_bytes(ctypes.byref(dims), ctypes.byref(out))
    if st != SOLO_OK:
        raise SoloError(st, "solo_readout_workspace_bytes")
    return out.value


def _ptr(t) -> int | None:
    if t is None:
        return None
    return t.data_ptr() if hasattr(t, "data_ptr") else int(t)


def _stream_handle(stream) -> int:
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _call(fn, dims, hidden, gamma, W, targets, mask, loss_tok, loss_mean, dhidden, dW, dgamma,
          workspace, workspace_bytes, stream, extra=()):
    K = dims.K
    if len(hidden) != K or len(dhidden) != K:
        raise ValueError("hidden and dhidden need K entries")
    harr = (ctypes.c_void_p * K)(*[_ptr(h) for h in hidden])
    darr = (ctypes.c_void_p * K)(*[_ptr(h) for h in dhidden])
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    st = fn(ctypes.byref(dims), harr, _ptr(gamma), _ptr(W), _ptr(targets), _ptr(mask),
            _ptr(loss_tok), _ptr(loss_mean), darr, _ptr(dW), _ptr(dgamma), _ptr(workspace),
            int(workspace_bytes), _stream_handle(stream), *extra)
    return st


def solo_readout_fwd_bwd(dims: solo_dims_t, hidden: Sequence, gamma, W, targets, mask,
                         loss_tok, loss_mean, dhidden: Sequence, dW, dgamma, workspace,
                         workspace_bytes: int | None = None, stream=None,
                         check: bool = True) -> int:
    """Enqueues one forward + backward; returns the status (raises on error when check)."""
    st = _call(load().solo_readout_fwd_bwd, dims, hidden, gamma, W, targets, mask, loss_tok,
               loss_mean, dhidden, dW, dgamma, workspace, workspace_bytes, stream)
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd")
    return st


def solo_readout_fwd_bwd_events(dims, hidden, gamma, W, targets, mask, loss_tok, loss_mean,
                                dhidden, dW, dgamma, workspace, events,
                                workspace_bytes: int | None = None, stream=None,
                                check: bool = True) -> int:
    """As solo_readout_fwd_bwd, recording ``events`` (SOLO_NUM_STAGES + 1 torch.cuda.Event
    with timing enabled) around the stages."""
    handles = []
    for e in events:
        h = e.cuda_event if hasattr(e, "cuda_event") else int(e)
        handles.append(h)
    arr = (ctypes.c_void_p * len(handles))(*handles)
    st = _call(load().solo_readout_fwd_bwd_events, dims, hidden, gamma, W, targets, mask,
               loss_tok, loss_mean, dhidden, dW, dgamma, workspace, workspace_bytes, stream,
               extra=(arr, len(handles)))
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd_events")
    return st


def solo_readout_fwd_bwd_static(dims: solo_dims_t, hidden: Sequence, gamma, W, targets, mask,
                                loss_tok, loss_mean, dhidden: Sequence, dW, dgamma,
                                device_flags=None, stream=None, check: bool = True) -> int:
    """The allocation-free variant: the library's built-in scratch replaces the
    workspace (problems up to SOLO_STATIC_SCRATCH_BYTES of scratch)."""
    K = dims.K
    if len(hidden) != K or len(dhidden) != K:
        raise ValueError("hidden and dhidden need K entries")
    harr = (ctypes.c_void_p * K)(*[_ptr(h) for h in hidden])
    darr = (ctypes.c_void_p * K)(*[_ptr(h) for h in dhidden])
    st = load().solo_readout_fwd_bwd_static(
        ctypes.byref(dims), harr, _ptr(gamma), _ptr(W), _ptr(targets), _ptr(mask),
        _ptr(loss_tok), _ptr(loss_mean), darr, _ptr(dW), _ptr(dgamma), _ptr(device_flags),
        _stream_handle(stream))
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd_static")
    return st


def solo_readout_exit_workspace_bytes(dims: solo_dims_t) -> int:
    out = ctypes.c_size_t(0)
    st = load().solo_readout_exit_workspace_bytes(ctypes.byref(dims), ctypes.byref(out))
    if st != SOLO_OK:
        raise SoloError(st, "solo_readout_exit_workspace_bytes")
    return out.value


def solo_readout_exit_forward(dims: solo_dims_t, hidden: Sequence, gamma, W, targets, mask,
                              loss_tok, loss_mean, top1, top1_logprob, workspace,
                              workspace_bytes: int | None = None, stream=None,
                              check: bool = True, events=None) -> int:
    """Early-exit readout (forward only): losses, top-1 and its log-probability per token.
    With ``events`` (SOLO_EXIT_NUM_STAGES + 1 torch.cuda.Event) the _events entry point
    is used and the stages are bracketed."""
    K = dims.K
    if len(hidden) != K:
        raise ValueError("hidden needs K entries")
    harr = (ctypes.c_void_p * K)(*[_ptr(h) for h in hidden])
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    args = [ctypes.byref(dims), harr, _ptr(gamma), _ptr(W), _ptr(targets), _ptr(mask),
            _ptr(loss_tok), _ptr(loss_mean), _ptr(top1), _ptr(top1_logprob), _ptr(workspace),
            int(workspace_bytes), _stream_handle(stream)]
    if events is None:
        st = load().solo_readout_exit_forward(*args)
        name = "solo_readout_exit_forward"
    else:
        handles = [e.cuda_event if hasattr(e, "cuda_event") else int(e) for e in events]
        arr = (ctypes.c_void_p * len(handles))(*handles)
        st = load().solo_readout_exit_forward_events(*args, arr, len(handles))
        name = "solo_readout_exit_forward_events"
    if check and st != SOLO_OK:
        raise SoloError(st, name)
    return st


class ExitReadout:
    """Owns the outputs and workspace of the early-exit readout for one size."""

    def __init__(self, K: int, N: int, d: int, V: int, eps: float = 1e-6,
                 ignore_index: int = -100, with_targets: bool = True, device=None):
        import torch
        self.dims = make_dims(K, N, d, V, eps, ignore_index)
        dev = torch.device("cuda" if device is None else device)
        self.workspace = torch.empty(solo_readout_exit_workspace_bytes(self.dims),
                                     dtype=torch.uint8, device=dev)
        self.loss_tok = torch.empty(K, N, dtype=torch.float32, device=dev) if with_targets else None
        self.loss_mean = torch.empty(K, dtype=torch.float32, device=dev) if with_targets else None
        self.top1 = torch.empty(K, N, dtype=torch.int32, device=dev)
        self.top1_logprob = torch.empty(K, N, dtype=torch.float32, device=dev)

    def __call__(self, hidden, gamma, W, targets=None, mask=None, stream=None, events=None):
        solo_readout_exit_forward(self.dims, hidden, gamma, W, targets, mask, self.loss_tok,
                                  self.loss_mean, self.top1, self.top1_logprob,
                                  self.workspace, stream=stream, events=events)
        return self

    def flags(self, stream=None) -> int:
        return solo_readout_get_flags(self.workspace, stream)


def solo_readout_fwd_bwd_heads(dims: solo_dims_t, hidden: Sequence, gamma, W, targets, mask,
                               tau, bias, dtau, dbias, loss_tok, loss_mean,
                               dhidden: Sequence, dW, dgamma, workspace,
                               workspace_bytes: int | None = None, stream=None, events=None,
                               check: bool = True) -> int:
    """The call with each head's temperature tau [K] and bias [K, V] (either may be None)."""
    K = dims.K
    if len(hidden) != K or len(dhidden) != K:
        raise ValueError("hidden and dhidden need K entries")
    harr = (ctypes.c_void_p * K)(*[_ptr(h) for h in hidden])
    darr = (ctypes.c_void_p * K)(*[_ptr(h) for h in dhidden])
    heads = solo_heads_t(_ptr(tau), _ptr(bias), _ptr(dtau), _ptr(dbias))
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    if events is None:
        earr, n = None, 0
    else:
        handles = [e.cuda_event if hasattr(e, "cuda_event") else int(e) for e in events]
        earr, n = (ctypes.c_void_p * len(handles))(*handles), len(handles)
    st = load().solo_readout_fwd_bwd_heads(
        ctypes.byref(dims), harr, _ptr(gamma), _ptr(W), _ptr(targets), _ptr(mask),
        ctypes.byref(heads), _ptr(loss_tok), _ptr(loss_mean), darr, _ptr(dW), _ptr(dgamma),
        _ptr(workspace), int(workspace_bytes), _stream_handle(stream), earr, n)
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd_heads")
    return st


def solo_readout_private_workspace_bytes(dims: solo_dims_t) -> int:
    out = ctypes.c_size_t(0)
    st = load().solo_readout_private_workspace_bytes(ctypes.byref(dims), ctypes.byref(out))
    if st != SOLO_OK:
        raise SoloError(st, "solo_readout_private_workspace_bytes")
    return out.value


def solo_readout_fwd_bwd_private(dims: solo_dims_t, hidden: Sequence, gammas: Sequence,
                                 Ws: Sequence, targets, mask, loss_tok, loss_mean,
                                 dhidden: Sequence, dWs, dgammas, workspace, tau=None, bias=None,
                                 dtau=None, dbias=None, workspace_bytes: int | None = None,
                                 stream=None, check: bool = True) -> int:
    """Private readouts W_k and head-owned gains gamma_k: dW_k and dgamma_k for every module."""
    K = dims.K
    arr = lambda xs: None if xs is None else (ctypes.c_void_p * K)(*[_ptr(x) for x in xs])
    heads = None
    if any(x is not None for x in (tau, bias, dtau, dbias)):
        heads = ctypes.byref(solo_heads_t(_ptr(tau), _ptr(bias), _ptr(dtau), _ptr(dbias)))
    if workspace_bytes is None:
        workspace_bytes = workspace.numel() * workspace.element_size()
    st = load().solo_readout_fwd_bwd_private(
        ctypes.byref(dims), arr(hidden), arr(gammas), arr(Ws), _ptr(targets), _ptr(mask), heads,
        _ptr(loss_tok), _ptr(loss_mean), arr(dhidden), arr(dWs), arr(dgammas), _ptr(workspace),
        int(workspace_bytes), _stream_handle(stream))
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd_private")
    return st


def solo_readout_onchip_workspace_bytes(dims: solo_dims_t) -> int:
    out = ctypes.c_size_t(0)
    st = load().solo_readout_onchip_workspace_bytes(ctypes.byref(dims), ctypes.byref(out))
    if st != SOLO_OK:
        raise SoloError(st, "solo_readout_onchip_workspace_bytes")
    return out.value


def solo_readout_fwd_bwd_onchip(dims: solo_dims_t, hidden: Sequence, gamma, W, targets, mask,
                                loss_tok, loss_mean, dhidden: Sequence, dW, dgamma, workspace,
                                workspace_bytes: int | None = None, stream=None, events=None,
                                check: bool = True) -> int:
    """The call with the auxiliary modules' logits kept on chip (events: None or
    SOLO_ONCHIP_NUM_STAGES + 1 torch.cuda.Event around its stages)."""
    if events is None:
        extra = (None, 0)
    else:
        handles = [e.cuda_event if hasattr(e, "cuda_event") else int(e) for e in events]
        extra = ((ctypes.c_void_p * len(handles))(*handles), len(handles))
    st = _call(load().solo_readout_fwd_bwd_onchip, dims, hidden, gamma, W, targets, mask,
               loss_tok, loss_mean, dhidden, dW, dgamma, workspace, workspace_bytes, stream,
               extra=extra)
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_fwd_bwd_onchip")
    return st


def solo_readout_get_flags(workspace, stream=None) -> int:
    out = ctypes.c_uint32(0)
    st = load().solo_readout_get_flags(_ptr(workspace), _stream_handle(stream), ctypes.byref(out))
    if st != SOLO_OK:
        raise SoloError(st, "solo_readout_get_flags")
    return out.value


def solo_readout_selftest_wait_timeout(device_flags, limit_us: int, stream=None,
                                       check: bool = True) -> int:
    """Runs the bounded-wait self-test; SOLO_FLAG_TIMEOUT lands in device_flags."""
    st = load().solo_readout_selftest_wait_timeout(_ptr(device_flags), int(limit_us),
                                                   _stream_handle(stream))
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_selftest_wait_timeout")
    return st


def solo_readout_version() -> int:
    return load().solo_readout_version()


def solo_readout_rmsnorm(dims: solo_dims_t, hidden: Sequence, gamma, xhat, r=None, stream=None,
                         check: bool = True) -> int:
    """The final RMSNorm alone: xhat bf16 [K*N, d] and, optionally, r fp32 [K*N]."""
    if len(hidden) != dims.K:
        raise ValueError("hidden needs K entries")
    harr = (ctypes.c_void_p * dims.K)(*[_ptr(h) for h in hidden])
    st = load().solo_readout_rmsnorm(ctypes.byref(dims), harr, _ptr(gamma), _ptr(xhat), _ptr(r),
                                     _stream_handle(stream))
    if check and st != SOLO_OK:
        raise SoloError(st, "solo_readout_rmsnorm")
    return st


def solo_readout_build_flags() -> int:
    """SOLO_BUILD_CHECKED (1) when the loaded library is the checked build."""
    return int(load().solo_readout_build_flags())


def solo_readout_kernel_launches() -> int:
    """Kernels the library has enqueued in this process so far."""
    return int(load().solo_readout_kernel_launches())


class Readout:
    """Owns the output and workspace tensors for one problem size (torch, one device).
    onchip=True selects solo_readout_fwd_bwd_onchip (the auxiliary modules' logits
    kept on chip) for calls without the heads' parameters."""

    def __init__(self, K: int, N: int, d: int, V: int, eps: float = 1e-6,
                 ignore_index: int = -100, want_loss_tok: bool = True, want_dW: bool = True,
                 want_dgamma: bool = True, device=None, onchip: bool = False):
        import torch
        self.dims = make_dims(K, N, d, V, eps, ignore_index)
        self.onchip = onchip
        dev = torch.device("cuda" if device is None else device)
        nbytes = (solo_readout_onchip_workspace_bytes(self.dims) if onchip
                  else solo_readout_workspace_bytes(self.dims))
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.loss_tok = torch.empty(K, N, dtype=torch.float32, device=dev) if want_loss_tok else None
        self.loss_mean = torch.empty(K, dtype=torch.float32, device=dev)
        self.dhidden = [torch.empty(N, d, dtype=torch.bfloat16, device=dev) for _ in range(K)]
        self.dW = torch.empty(V, d, dtype=torch.float32, device=dev) if want_dW else None
        self.dgamma = torch.empty(d, dtype=torch.float32, device=dev) if want_dgamma else None
        self.dtau = torch.empty(K, dtype=torch.float32, device=dev)
        self.dbias = torch.empty(K, V, dtype=torch.float32, device=dev)

    def __call__(self, hidden, gamma, W, targets, mask=None, stream=None, events=None,
                 tau=None, bias=None, head_grads=False):
        """tau [K] / bias [K, V] (fp32, either may be None) select the heads' call;
        head_grads also fills self.dtau and self.dbias."""
        if self.onchip:
            if tau is not None or bias is not None or head_grads:
                raise ValueError("the on-chip call takes no heads' parameters")
            solo_readout_fwd_bwd_onchip(self.dims, hidden, gamma, W, targets, mask,
                                        self.loss_tok, self.loss_mean, self.dhidden, self.dW,
                                        self.dgamma, self.workspace, stream=stream,
                                        events=events)
        elif tau is not None or bias is not None or head_grads:
            solo_readout_fwd_bwd_heads(self.dims, hidden, gamma, W, targets, mask, tau, bias,
                                       self.dtau if head_grads else None,
                                       self.dbias if head_grads else None, self.loss_tok,
                                       self.loss_mean, self.dhidden, self.dW, self.dgamma,
                                       self.workspace, stream=stream, events=events)
        elif events is None:
            solo_readout_fwd_bwd(self.dims, hidden, gamma, W, targets, mask, self.loss_tok,
                                 self.loss_mean, self.dhidden, self.dW, self.dgamma,
                                 self.workspace, stream=stream)
        else:
            solo_readout_fwd_bwd_events(self.dims, hidden, gamma, W, targets, mask,
                                        self.loss_tok, self.loss_mean, self.dhidden, self.dW,
                                        self.dgamma, self.workspace, events, stream=stream)
        return self

    def flags(self, stream=None) -> int:
        return solo_readout_get_flags(self.workspace, stream)
