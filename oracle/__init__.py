"""Float64 CPU oracle for the OPD reverse-KL step (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline and
``--impl reference`` legs may import this package. The CUDA library never
loads it, and it shares no code with the library: the arithmetic lives in
``opd_kl_oracle.cpp`` (plain loops, materialised logits, two-pass log-softmax),
this file only compiles it with g++ and marshals numpy arrays through ctypes.

Definitions followed: ActFirst-OPD Section 3, Eq. opd-objective and
Eq. reverse-kl (per-token reverse KL over the full vocabulary); Appendix B.4
(mask m = 1 on model-generated response tokens, frozen teacher,
seq-mean-token-mean aggregation with eps = 1e-8).
"""

from __future__ import annotations

import ctypes
import os
import subprocess
from dataclasses import dataclass
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "opd_kl_oracle.cpp")
_LIB = os.path.join(_HERE, "_build", "libopd_oracle.so")
_lib = None

KIND_F32 = 0
KIND_BF16 = 1


def build(force: bool = False) -> str:
    """Compile the oracle with g++ (no fast-math, no FMA contraction)."""
    os.makedirs(os.path.dirname(_LIB), exist_ok=True)
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + f".tmp{os.getpid()}"
    cmd = ["g++", "-O2", "-std=c++17", "-ffp-contract=off", "-fno-fast-math", "-shared",
           "-fPIC", "-pthread", _SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        p = ctypes.c_void_p
        i64 = ctypes.c_int64
        lib.opd_oracle_kl.argtypes = [i64, i64, i64, i64, ctypes.c_double, ctypes.c_int,
                                      p, p, p, p, p, p, p, i64, p, p, p, p, p, p, ctypes.c_int]
        lib.opd_oracle_kl.restype = ctypes.c_int
        lib.opd_oracle_seq_mean_token_mean_weights.argtypes = [p, p, i64, ctypes.c_double, p]
        lib.opd_oracle_seq_mean_token_mean_weights.restype = ctypes.c_int
        dbl = ctypes.c_double
        lib.opd_oracle_score.argtypes = [i64, i64, i64, dbl, ctypes.c_int, p, p, p, p, i64, p, p, ctypes.c_int]
        lib.opd_oracle_score.restype = ctypes.c_int
        lib.opd_oracle_surrogate.argtypes = [i64, i64, i64, dbl, ctypes.c_int, p, p, p, p, p, p, p, dbl, dbl, dbl,
                                             p, i64, p, p, p, p, p, p, ctypes.c_int]
        lib.opd_oracle_surrogate.restype = ctypes.c_int
        lib.opd_oracle_dual_clip.argtypes = [i64, p, p, p, dbl, dbl, dbl, p, p]
        lib.opd_oracle_dual_clip.restype = ctypes.c_int
        _lib = lib
    return _lib


def _ptr(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _as_input(a: np.ndarray):
    """Accept float32 values or bf16 bit patterns (uint16); anything else is widened to float32."""
    if a.dtype == np.uint16:
        return np.ascontiguousarray(a), KIND_BF16
    return np.ascontiguousarray(a, dtype=np.float32), KIND_F32


@dataclass
class OracleResult:
    kl: np.ndarray
    lse_s: np.ndarray
    lse_t: np.ndarray
    dZ: Optional[np.ndarray]
    dH_s: Optional[np.ndarray]
    dW_s: Optional[np.ndarray]


def default_threads() -> int:
    return max(1, os.cpu_count() or 1)


def opd_kl(H_s, H_t, W_s, W_t, mask, g, tau: float = 1.0, rows=None, want_dZ: bool = False,
           want_dH: bool = True, want_dW: bool = True, n_threads: Optional[int] = None) -> OracleResult:
    """Per-token reverse KL and its gradient, in float64.

    H_s [T, d_s], H_t [T, d_t], W_s [V, d_s], W_t [V, d_t]: float32, or uint16 bf16 bit
    patterns (all four the same kind). mask [T] (nonzero = supervised), g [T] upstream
    weights dL/dKL_i. ``rows``: indices to evaluate (default all T); outputs follow that
    list, except dW_s [V, d_s], the sum over the listed rows.
    """
    lib = _load()
    Hs, kind = _as_input(H_s)
    Ht, k2 = _as_input(H_t)
    Ws, k3 = _as_input(W_s)
    Wt, k4 = _as_input(W_t)
    if len({kind, k2, k3, k4}) != 1:
        raise ValueError("H_s, H_t, W_s, W_t must share one element kind")
    T, d_s = Hs.shape
    T2, d_t = Ht.shape
    V = Ws.shape[0]
    if T2 != T or Ws.shape != (V, d_s) or Wt.shape != (V, d_t):
        raise ValueError("shape mismatch")
    m = np.ascontiguousarray(np.asarray(mask) != 0, dtype=np.uint8)
    gg = np.ascontiguousarray(g, dtype=np.float64)
    if m.shape != (T,) or gg.shape != (T,):
        raise ValueError("mask and g must have shape [T]")
    r = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    n = T if r is None else r.shape[0]
    kl = np.zeros(n)
    lse_s = np.zeros(n)
    lse_t = np.zeros(n)
    dZ = np.zeros((n, V)) if want_dZ else None
    dH = np.zeros((n, d_s)) if want_dH else None
    dW = np.zeros((V, d_s)) if want_dW else None
    rc = lib.opd_oracle_kl(T, d_s, d_t, V, float(tau), kind, _ptr(Hs), _ptr(Ht), _ptr(Ws), _ptr(Wt),
                           _ptr(m), _ptr(gg), _ptr(r), n, _ptr(kl), _ptr(lse_s), _ptr(lse_t),
                           _ptr(dZ), _ptr(dH), _ptr(dW), int(n_threads or default_threads()))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return OracleResult(kl, lse_s, lse_t, dZ, dH, dW)


def seq_mean_token_mean_weights(seg_id, mask, eps: float = 1e-8) -> np.ndarray:
    """dL/dKL_i for L = seq-mean-token-mean of per-token losses (Appendix B.4, Eq. opd-surrogate)."""
    lib = _load()
    s = np.ascontiguousarray(seg_id, dtype=np.int32)
    m = np.ascontiguousarray(np.asarray(mask) != 0, dtype=np.uint8)
    w = np.zeros(s.shape[0])
    rc = lib.opd_oracle_seq_mean_token_mean_weights(_ptr(s), _ptr(m), s.shape[0], float(eps), _ptr(w))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return w


# Constants of the surrogate (Appendix B.4): clipping width, dual-clip constant, log-ratio clip.
DELTA = 0.2
KAPPA = 3.0
LOG_RATIO_CLIP = 20.0


def score(H, W, tokens, tau: float = 1.0, rows=None, n_threads: Optional[int] = None):
    """(lse, logp) of the given tokens under one head, float64, for every listed row."""
    lib = _load()
    Hh, kind = _as_input(H)
    Wh, k2 = _as_input(W)
    if kind != k2:
        raise ValueError("H and W must share one element kind")
    T, d = Hh.shape
    V = Wh.shape[0]
    if Wh.shape != (V, d):
        raise ValueError("shape mismatch")
    tok = np.ascontiguousarray(tokens, dtype=np.int32)
    r = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    n = T if r is None else r.shape[0]
    lse = np.zeros(n)
    logp = np.zeros(n)
    rc = lib.opd_oracle_score(T, d, V, float(tau), kind, _ptr(Hh), _ptr(Wh), _ptr(tok), _ptr(r), n, _ptr(lse),
                              _ptr(logp), int(n_threads or default_threads()))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return lse, logp


@dataclass
class SurrogateResult:
    loss: np.ndarray
    logp_s: np.ndarray
    adv: np.ndarray
    dZ: Optional[np.ndarray]
    dH_s: Optional[np.ndarray]
    dW_s: Optional[np.ndarray]


def surrogate(H_s, W_s, tokens, logp_old, logp_teacher, mask, w, tau: float = 1.0, delta: float = DELTA,
              kappa: float = KAPPA, clip: float = LOG_RATIO_CLIP, rows=None, want_dZ: bool = False,
              want_dH: bool = True, want_dW: bool = True, n_threads: Optional[int] = None) -> SurrogateResult:
    """Sampled-token dual-clip surrogate (student side) and its gradient, float64."""
    lib = _load()
    Hh, kind = _as_input(H_s)
    Wh, k2 = _as_input(W_s)
    if kind != k2:
        raise ValueError("H_s and W_s must share one element kind")
    T, d = Hh.shape
    V = Wh.shape[0]
    if Wh.shape != (V, d):
        raise ValueError("shape mismatch")
    tok = np.ascontiguousarray(tokens, dtype=np.int32)
    lo = np.ascontiguousarray(logp_old, dtype=np.float64)
    lt = np.ascontiguousarray(logp_teacher, dtype=np.float64)
    m = np.ascontiguousarray(np.asarray(mask) != 0, dtype=np.uint8)
    ww = np.ascontiguousarray(w, dtype=np.float64)
    for a in (tok, lo, lt, m, ww):
        if a.shape != (T,):
            raise ValueError("per-token inputs must have shape [T]")
    r = None if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    n = T if r is None else r.shape[0]
    loss, lps, adv = np.zeros(n), np.zeros(n), np.zeros(n)
    dZ = np.zeros((n, V)) if want_dZ else None
    dH = np.zeros((n, d)) if want_dH else None
    dW = np.zeros((V, d)) if want_dW else None
    rc = lib.opd_oracle_surrogate(T, d, V, float(tau), kind, _ptr(Hh), _ptr(Wh), _ptr(tok), _ptr(lo), _ptr(lt),
                                  _ptr(m), _ptr(ww), float(delta), float(kappa), float(clip), _ptr(r), n,
                                  _ptr(loss), _ptr(lps), _ptr(adv), _ptr(dZ), _ptr(dH), _ptr(dW),
                                  int(n_threads or default_threads()))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return SurrogateResult(loss, lps, adv, dZ, dH, dW)


def dual_clip(logp_s, logp_old, A, delta: float = DELTA, kappa: float = KAPPA, clip: float = LOG_RATIO_CLIP):
    """Per-token dual-clip loss and d loss / d logp_s (elementwise)."""
    lib = _load()
    a = np.ascontiguousarray(logp_s, dtype=np.float64)
    b = np.ascontiguousarray(logp_old, dtype=np.float64)
    c = np.ascontiguousarray(A, dtype=np.float64)
    loss, dl = np.zeros(a.shape[0]), np.zeros(a.shape[0])
    rc = lib.opd_oracle_dual_clip(a.shape[0], _ptr(a), _ptr(b), _ptr(c), float(delta), float(kappa), float(clip),
                                  _ptr(loss), _ptr(dl))
    if rc != 0:
        raise ValueError("oracle rejected its arguments")
    return loss, dl
