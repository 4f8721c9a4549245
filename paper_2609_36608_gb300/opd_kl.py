"""Python binding of the C ABI in include/opd_kl.h (ctypes, argument marshalling only).

Every function has the C entry point's name and forwards to it: all of the
computation runs in the CUDA library libopdkl.so. PyTorch supplies device
memory and streams. There is no fallback: importing this module fails loudly
when the library has not been built (``python -m paper_2609_36608_gb300.build``).
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import numpy as np
import torch

from . import build as _build

OPD_OK = 0
OPD_ERR_INVALID_ARG = 1
OPD_ERR_UNSUPPORTED = 2
OPD_ERR_CUDA = 3
OPD_ERR_TIMEOUT = 4
OPD_ERR_NONFINITE = 5

OPD_DTYPE_BF16 = 0
OPD_DTYPE_F32 = 1

OPD_KL_NOALLOC_MAX_ROWS = 4096


class opd_problem(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int64), ("d_s", ctypes.c_int64), ("d_t", ctypes.c_int64), ("V", ctypes.c_int64),
                ("dtype", ctypes.c_int32), ("temperature", ctypes.c_float)]


class opd_kernel_time(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_int64), ("total_ms", ctypes.c_double)]


class opd_surrogate_params(ctypes.Structure):
    _fields_ = [("delta", ctypes.c_float), ("kappa", ctypes.c_float), ("log_ratio_clip", ctypes.c_float)]


class OpdError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: {opd_status_string(status)} ({status})")
        self.status = status


def _load() -> ctypes.CDLL:
    path = _build.LIB
    if not os.path.exists(path):
        raise RuntimeError(f"libopdkl.so is not built ({path}); run python -m paper_2609_36608_gb300.build")
    lib = ctypes.CDLL(path)
    P = ctypes.POINTER(opd_problem)
    vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_size_t
    sig = {
        "opd_kl_workspace_size": (sz, [P]),
        "opd_kl_forward_workspace_size": (sz, [P]),
        "opd_kl_forward": (i32, [P, vp, vp, vp, vp, vp, vp, vp, vp, sz, vp]),
        "opd_kl_forward_noalloc": (i32, [P, vp, vp, vp, vp, vp, vp, vp, vp]),
        "opd_kl_backward": (i32, [P, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32, vp, sz, vp]),
        "opd_kl_fwd_bwd": (i32, [P, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, i32, vp, sz, vp]),
        "opd_seq_mean_token_mean_weights": (i32, [vp, vp, i64, ctypes.c_float, vp]),
        "opd_kl_get_status": (i32, [vp, sz, vp]),
        "opd_kl_selftest_timeout": (i32, [vp, sz, ctypes.c_uint64, vp]),
        "opd_status_string": (ctypes.c_char_p, [i32]),
        "opd_score_tokens": (i32, [P, vp, vp, vp, vp, vp, vp, vp, sz, vp]),
        "opd_surrogate_fwd_bwd": (i32, [P, vp, vp, vp, vp, vp, vp, vp, ctypes.POINTER(opd_surrogate_params),
                                        vp, vp, vp, vp, i32, vp, sz, vp]),
        "opd_seq_mean_token_mean_workspace_size": (sz, [i64]),
        "opd_kl_seq_mean_workspace_size": (sz, [P, i64]),
        "opd_kl_seq_mean_fwd_bwd": (i32, [P, vp, vp, vp, vp, vp, vp, i64, ctypes.c_float, vp, vp, vp, vp, vp, i32,
                                          vp, sz, vp]),
        "opd_seq_mean_token_mean_device": (i32, [vp, vp, i64, i64, ctypes.c_float, vp, vp, vp, vp, sz, vp]),
        "opd_seq_mean_token_mean_counts": (i32, [vp, vp, i64, i64, vp, vp, sz, vp]),
        "opd_seq_mean_token_mean_from_counts": (i32, [vp, vp, i64, i64, vp, ctypes.c_float, vp, vp, vp, vp, sz,
                                                      vp]),
        "opd_kl_profile_start": (i32, []),
        "opd_kl_profile_stop": (i32, [ctypes.POINTER(opd_kernel_time), i32, ctypes.POINTER(i32)]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()
LIBRARY_PATH = _build.LIB


def opd_status_string(status: int) -> str:
    return _lib.opd_status_string(int(status)).decode()


def make_problem(T: int, d_s: int, d_t: int, V: int, dtype: int = OPD_DTYPE_BF16,
                 temperature: float = 1.0) -> opd_problem:
    return opd_problem(int(T), int(d_s), int(d_t), int(V), int(dtype), float(temperature))


_F32 = (torch.float32,)
_I32 = (torch.int32,)
_BYTE = (torch.uint8, torch.bool)  # one byte per row, nonzero = supervised


class _Buffers:
    """Device pointers of the buffers one call reads or writes.

    The library sees only the pointers, so every buffer is checked here against what the
    call will touch: a contiguous tensor of the element type the C signature documents,
    holding at least `numel` elements; then, once every buffer has passed that, a CUDA
    tensor on the current device. A wrong buffer raises before any launch instead of
    reaching a kernel. None passes through as NULL (the C entry points reject a NULL
    they need)."""

    def __init__(self):
        self.seen = []

    def __call__(self, t: Optional[torch.Tensor], name: str, dtypes=None, numel: int = 0):
        if t is None:
            return None
        if not isinstance(t, torch.Tensor):
            raise TypeError(f"{name}: expected a torch.Tensor")
        if dtypes is not None and t.dtype not in dtypes:
            raise TypeError(f"{name}: dtype {t.dtype}, expected {' or '.join(str(d) for d in dtypes)}")
        if not t.is_contiguous():
            raise ValueError(f"{name}: buffers must be contiguous")
        if t.numel() < numel:
            raise ValueError(f"{name} holds {t.numel()} elements; the problem needs {numel}")
        self.seen.append((name, t))
        return ctypes.c_void_p(t.data_ptr()) if t.numel() > 0 else None

    def on_device(self) -> None:
        for name, t in self.seen:
            if not t.is_cuda:
                raise ValueError(f"{name}: device buffers must be CUDA tensors")
            if t.device.index != torch.cuda.current_device():
                raise ValueError(f"{name} is on {t.device}, but the current device is "
                                 f"cuda:{torch.cuda.current_device()}")


def _nbytes(t: Optional[torch.Tensor]) -> int:
    return 0 if t is None else t.numel() * t.element_size()


def _inputs(problem) -> tuple:
    return (torch.bfloat16,) if problem.dtype == OPD_DTYPE_BF16 else (torch.float32,)


def _kl_inputs(b: _Buffers, problem, H_s, H_t, W_s, W_t, mask) -> list:
    T, ds, dt, V, x = problem.T, problem.d_s, problem.d_t, problem.V, _inputs(problem)
    return [b(H_s, "H_s", x, T * ds), b(H_t, "H_t", x, T * dt), b(W_s, "W_s", x, V * ds), b(W_t, "W_t", x, V * dt),
            b(mask, "mask", _BYTE, T)]


def _call(name: str, b: _Buffers, args: list, stream) -> int:
    """Checks the buffers' device, then calls the entry point with the stream appended."""
    b.on_device()
    return int(getattr(_lib, name)(*args, _stream(stream)))


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    if isinstance(stream, torch.cuda.Stream):
        stream = stream.cuda_stream
    return ctypes.c_void_p(int(stream))


def _check(status: int, what: str) -> None:
    if status != OPD_OK:
        raise OpdError(status, what)


def opd_kl_workspace_size(problem: opd_problem) -> int:
    return int(_lib.opd_kl_workspace_size(ctypes.byref(problem)))


def opd_kl_forward_workspace_size(problem: opd_problem) -> int:
    return int(_lib.opd_kl_forward_workspace_size(ctypes.byref(problem)))


def allocate_workspace(problem: opd_problem, device="cuda", forward_only: bool = False) -> torch.Tensor:
    """A workspace for every call on this problem, or (forward_only) the smaller one that
    opd_kl_forward and opd_score_tokens need."""
    n = opd_kl_forward_workspace_size(problem) if forward_only else opd_kl_workspace_size(problem)
    if n == 0:
        raise ValueError("invalid problem")
    return torch.empty(n, dtype=torch.uint8, device=device)


def opd_kl_forward(problem, H_s, H_t, W_s, W_t, mask, kl_out, stats, workspace, stream=None) -> None:
    T, b = problem.T, _Buffers()
    args = [ctypes.byref(problem), *_kl_inputs(b, problem, H_s, H_t, W_s, W_t, mask),
            b(kl_out, "kl_out", _F32, T), b(stats, "stats", _F32, 3 * T),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_kl_forward", b, args, stream), "opd_kl_forward")


def opd_kl_forward_noalloc(problem, H_s, H_t, W_s, W_t, mask, kl_out, stats, stream=None) -> None:
    """opd_kl_forward without a workspace, for callers that may not allocate device memory
    (T <= OPD_KL_NOALLOC_MAX_ROWS, bf16; scratch is a fixed array inside the library)."""
    T, b = problem.T, _Buffers()
    args = [ctypes.byref(problem), *_kl_inputs(b, problem, H_s, H_t, W_s, W_t, mask),
            b(kl_out, "kl_out", _F32, T), b(stats, "stats", _F32, 3 * T)]
    _check(_call("opd_kl_forward_noalloc", b, args, stream), "opd_kl_forward_noalloc")


def opd_kl_backward(problem, H_s, H_t, W_s, W_t, mask, stats, grad_kl, dH_s, dW_s, accumulate_dW: bool,
                    workspace, stream=None) -> None:
    T, ds, V, b = problem.T, problem.d_s, problem.V, _Buffers()
    args = [ctypes.byref(problem), *_kl_inputs(b, problem, H_s, H_t, W_s, W_t, mask),
            b(stats, "stats", _F32, 3 * T), b(grad_kl, "grad_kl", _F32, T), b(dH_s, "dH_s", _F32, T * ds),
            b(dW_s, "dW_s", _F32, V * ds), int(bool(accumulate_dW)),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_kl_backward", b, args, stream), "opd_kl_backward")


def opd_kl_fwd_bwd(problem, H_s, H_t, W_s, W_t, mask, grad_kl, kl_out, stats, dH_s, dW_s, accumulate_dW: bool,
                   workspace, stream=None) -> None:
    T, ds, V, b = problem.T, problem.d_s, problem.V, _Buffers()
    args = [ctypes.byref(problem), *_kl_inputs(b, problem, H_s, H_t, W_s, W_t, mask),
            b(grad_kl, "grad_kl", _F32, T), b(kl_out, "kl_out", _F32, T), b(stats, "stats", _F32, 3 * T),
            b(dH_s, "dH_s", _F32, T * ds), b(dW_s, "dW_s", _F32, V * ds), int(bool(accumulate_dW)),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_kl_fwd_bwd", b, args, stream), "opd_kl_fwd_bwd")


def opd_kl_seq_mean_workspace_size(problem, n_ids: int) -> int:
    return int(_lib.opd_kl_seq_mean_workspace_size(ctypes.byref(problem), int(n_ids)))


def allocate_seq_mean_workspace(problem, n_ids: int, device="cuda") -> torch.Tensor:
    n = opd_kl_seq_mean_workspace_size(problem, n_ids)
    if n == 0:
        raise ValueError("invalid problem or n_ids")
    return torch.empty(n, dtype=torch.uint8, device=device)


def opd_kl_seq_mean_fwd_bwd(problem, H_s, H_t, W_s, W_t, mask, seg_id, n_ids: int, eps: float, loss_out, kl_out,
                            stats, dH_s, dW_s, accumulate_dW: bool, workspace, stream=None) -> None:
    """The paper's batch loss over the per-token KL (seq-mean-token-mean weights on the device, L summed
    in the combine pass) and its gradients, in one call."""
    T, ds, V, b = problem.T, problem.d_s, problem.V, _Buffers()
    args = [ctypes.byref(problem), *_kl_inputs(b, problem, H_s, H_t, W_s, W_t, mask),
            b(seg_id, "seg_id", _I32, T), int(n_ids), float(eps), b(loss_out, "loss_out", _F32, 1),
            b(kl_out, "kl_out", _F32, T), b(stats, "stats", _F32, 3 * T), b(dH_s, "dH_s", _F32, T * ds),
            b(dW_s, "dW_s", _F32, V * ds), int(bool(accumulate_dW)),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_kl_seq_mean_fwd_bwd", b, args, stream), "opd_kl_seq_mean_fwd_bwd")


def opd_score_tokens(problem, H, W, tokens, mask, lse_out, logp_out, workspace, stream=None) -> None:
    """Log-partition and log-probability of the given tokens under one head (d = problem.d_s)."""
    T, d, V, x, b = problem.T, problem.d_s, problem.V, _inputs(problem), _Buffers()
    args = [ctypes.byref(problem), b(H, "H", x, T * d), b(W, "W", x, V * d), b(tokens, "tokens", _I32, T),
            b(mask, "mask", _BYTE, T), b(lse_out, "lse_out", _F32, T), b(logp_out, "logp_out", _F32, T),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_score_tokens", b, args, stream), "opd_score_tokens")


def opd_surrogate_fwd_bwd(problem, H_s, W_s, tokens, logp_old, logp_teacher, mask, weights, loss_out, logp_out,
                          dH_s, dW_s, accumulate_dW: bool, workspace, params=None, stream=None) -> None:
    """Sampled-token dual-clip surrogate, forward and backward (student side)."""
    T, d, V, x, b = problem.T, problem.d_s, problem.V, _inputs(problem), _Buffers()
    pp = ctypes.byref(params) if params is not None else None
    args = [ctypes.byref(problem), b(H_s, "H_s", x, T * d), b(W_s, "W_s", x, V * d), b(tokens, "tokens", _I32, T),
            b(logp_old, "logp_old", _F32, T), b(logp_teacher, "logp_teacher", _F32, T), b(mask, "mask", _BYTE, T),
            b(weights, "weights", _F32, T), pp, b(loss_out, "loss_out", _F32, T), b(logp_out, "logp_out", _F32, T),
            b(dH_s, "dH_s", _F32, T * d), b(dW_s, "dW_s", _F32, V * d), int(bool(accumulate_dW)),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_surrogate_fwd_bwd", b, args, stream), "opd_surrogate_fwd_bwd")


def opd_seq_mean_token_mean_weights(seg_id, mask, eps: float = 1e-8) -> np.ndarray:
    s = np.ascontiguousarray(seg_id, dtype=np.int32)
    m = np.ascontiguousarray(np.asarray(mask) != 0, dtype=np.uint8)
    w = np.zeros(s.shape[0], dtype=np.float32)
    _check(_lib.opd_seq_mean_token_mean_weights(s.ctypes.data_as(ctypes.c_void_p), m.ctypes.data_as(ctypes.c_void_p),
                                                s.shape[0], float(eps), w.ctypes.data_as(ctypes.c_void_p)),
           "opd_seq_mean_token_mean_weights")
    return w


def opd_seq_mean_token_mean_workspace_size(n_ids: int) -> int:
    return int(_lib.opd_seq_mean_token_mean_workspace_size(int(n_ids)))


def opd_seq_mean_token_mean_device(seg_id, mask, n_ids: int, eps: float = 1e-8, loss_in=None, w_out=None,
                                   loss_out=None, workspace=None, stream=None) -> torch.Tensor:
    """seq-mean-token-mean weights (and optionally the weighted loss) on the device; returns the
    workspace used (its status word is what opd_kl_get_status reads)."""
    if workspace is None:
        workspace = torch.empty(opd_seq_mean_token_mean_workspace_size(n_ids), dtype=torch.uint8,
                                device=seg_id.device)
    T, b = seg_id.numel(), _Buffers()
    args = [b(seg_id, "seg_id", _I32, T), b(mask, "mask", _BYTE, T), T, int(n_ids), float(eps),
            b(loss_in, "loss_in", _F32, T), b(w_out, "w_out", _F32, T), b(loss_out, "loss_out", _F32, 1),
            b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_seq_mean_token_mean_device", b, args, stream), "opd_seq_mean_token_mean_device")
    return workspace


def opd_seq_mean_token_mean_counts(seg_id, mask, n_ids: int, counts, workspace, stream=None) -> None:
    """This process's rows per response id: counts [2, n_ids] int32 (supervised rows, all rows)."""
    T, b = seg_id.numel(), _Buffers()
    args = [b(seg_id, "seg_id", _I32, T), b(mask, "mask", _BYTE, T), T, int(n_ids),
            b(counts, "counts", _I32, 2 * int(n_ids)), b(workspace, "workspace"), _nbytes(workspace)]
    _check(_call("opd_seq_mean_token_mean_counts", b, args, stream), "opd_seq_mean_token_mean_counts")


def opd_seq_mean_token_mean_from_counts(seg_id, mask, n_ids: int, counts, eps: float = 1e-8, loss_in=None,
                                        w_out=None, loss_out=None, workspace=None, stream=None) -> None:
    """seq-mean-token-mean weights of this process's rows (and its part of the batch loss) from
    the per-id counts summed over every process."""
    T, b = seg_id.numel(), _Buffers()
    args = [b(seg_id, "seg_id", _I32, T), b(mask, "mask", _BYTE, T), T, int(n_ids),
            b(counts, "counts", _I32, 2 * int(n_ids)), float(eps), b(loss_in, "loss_in", _F32, T),
            b(w_out, "w_out", _F32, T), b(loss_out, "loss_out", _F32, 1), b(workspace, "workspace"),
            _nbytes(workspace)]
    _check(_call("opd_seq_mean_token_mean_from_counts", b, args, stream), "opd_seq_mean_token_mean_from_counts")


def opd_kl_get_status(workspace, stream=None) -> int:
    b = _Buffers()
    return _call("opd_kl_get_status", b, [b(workspace, "workspace"), _nbytes(workspace)], stream)


def opd_kl_selftest_timeout(workspace, limit_ns: int, stream=None) -> int:
    b = _Buffers()
    return _call("opd_kl_selftest_timeout", b, [b(workspace, "workspace"), _nbytes(workspace), int(limit_ns)],
                 stream)


def opd_kl_profile_start() -> None:
    _check(_lib.opd_kl_profile_start(), "opd_kl_profile_start")


def opd_kl_profile_stop() -> dict:
    """{kernel name: (launches, total event milliseconds)} since opd_kl_profile_start."""
    cap = 64
    buf = (opd_kernel_time * cap)()
    n = ctypes.c_int(0)
    _check(_lib.opd_kl_profile_stop(buf, cap, ctypes.byref(n)), "opd_kl_profile_stop")
    return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms)) for i in range(min(n.value, cap))}


def call_raw(name: str, *args) -> int:
    """Call an entry point with raw ctypes arguments (argument-validation tests)."""
    return int(getattr(_lib, name)(*args))
