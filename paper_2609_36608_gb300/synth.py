"""Seeded synthetic workloads for the OPD reverse-KL step.

This module is the one piece shared by the CUDA path's tests/benchmark and the
CPU oracle's tests: it draws inputs and nothing else. It holds none of the
method's arithmetic (no logits, softmax, KL or gradients).

Random numbers come from a counter-based generator: the PCG hash of
Jarzynski and Olano ("Hash Functions for GPU Rendering", JCGT 2020), applied
twice, with the element index as counter and a per-tensor key. Normal variates
use the Box-Muller transform (Box and Muller, 1958) in float64, then round to
float32 and, for bf16 workloads, to bf16 (round to nearest even, torch's cast).
All integer steps stay below 2**63, so the same code runs on CPU and GPU tensors.

Workload shapes follow the paper's training setup: packed multi-turn batches of
turn-level responses (Appendix C, 16,384-token dynamic-batching budget per GPU;
512-token response limit with a 384-token first thinking stage), masked
observation/prompt tokens, and masked inserted thinking-budget tokens inside a
response (Appendix B.3 "Thinking Budget", Appendix B.4 mask m).
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Dict, List, Optional, Tuple

import numpy as np
import torch

_M32 = 0xFFFFFFFF

# Tensor stream ids (part of the per-tensor key).
STREAM_H_S, STREAM_H_T, STREAM_W_S, STREAM_W_T = 1, 2, 3, 4
STREAM_H_T_EXTRA, STREAM_W_T_EXTRA = 5, 6
STREAM_LAYOUT = 7
STREAM_G = 8
STREAM_TOKENS = 9


def pcg_hash_int(x: int) -> int:
    """PCG-RXS-M-XS 32-bit hash on a Python int in [0, 2**32)."""
    state = (x * 747796405 + 2891336453) & _M32
    word = (((state >> ((state >> 28) + 4)) ^ state) * 277803737) & _M32
    return ((word >> 22) ^ word) & _M32


def _pcg_hash(x: torch.Tensor) -> torch.Tensor:
    """The same hash elementwise on an int64 tensor with values in [0, 2**32)."""
    state = (x * 747796405 + 2891336453) & _M32
    word = (((state >> ((state >> 28) + 4)) ^ state) * 277803737) & _M32
    return ((word >> 22) ^ word) & _M32


def stream_key(seed: int, stream: int) -> int:
    return pcg_hash_int((pcg_hash_int(seed & _M32) + 0x9E3779B9 * stream) & _M32)


def uniform_bits(key: int, start: int, count: int, device) -> torch.Tensor:
    """32-bit draws for counters start .. start+count-1 (int64 tensor)."""
    n = torch.arange(start, start + count, dtype=torch.int64, device=device)
    return _pcg_hash(_pcg_hash(n) ^ key)


def normal(seed: int, stream: int, numel: int, device="cpu") -> torch.Tensor:
    """numel standard normal draws (float64); elements 2p and 2p+1 share one Box-Muller pair."""
    return _normal_range(seed, stream, 0, numel, device)


def normal_tensor(seed: int, stream: int, shape: Tuple[int, ...], std: float, dtype: torch.dtype,
                  device="cpu") -> torch.Tensor:
    """N(0, std^2) draws rounded float64 -> float32 -> dtype."""
    numel = int(np.prod(shape))
    out = torch.empty(shape, dtype=dtype, device=device)
    flat = out.view(-1)
    block = 1 << 26
    # Generate in blocks so the float64 temporaries stay bounded; the counter
    # space is global to the tensor, so blocking does not change the values.
    for lo in range(0, numel, block):
        hi = min(lo + block, numel)
        z = _normal_range(seed, stream, lo, hi, device)
        flat[lo:hi] = (z * std).to(torch.float32).to(dtype)
    return out


def _normal_range(seed: int, stream: int, lo: int, hi: int, device) -> torch.Tensor:
    key = stream_key(seed, stream)
    plo = lo - (lo & 1)
    phi = hi + (hi & 1)
    bits = uniform_bits(key, plo, phi - plo, device)
    u1 = (bits[0::2].to(torch.float64) + 0.5) * (2.0 ** -32)
    u2 = bits[1::2].to(torch.float64) * (2.0 ** -32)
    r = torch.sqrt(-2.0 * torch.log(u1))
    theta = (2.0 * math.pi) * u2
    z = torch.empty(phi - plo, dtype=torch.float64, device=device)
    z[0::2] = r * torch.cos(theta)
    z[1::2] = r * torch.sin(theta)
    return z[lo - plo:lo - plo + (hi - lo)]


class Draws:
    """Sequential scalar draws from one counter stream (for layouts)."""

    def __init__(self, seed: int, stream: int):
        self.key = stream_key(seed, stream)
        self.n = 0

    def bits(self) -> int:
        b = pcg_hash_int(pcg_hash_int(self.n & _M32) ^ self.key)
        self.n += 1
        return b

    def uniform(self) -> float:
        return (self.bits() + 0.5) * (2.0 ** -32)

    def randint(self, lo: int, hi: int) -> int:
        """Uniform integer in [lo, hi] inclusive."""
        span = hi - lo + 1
        return lo + min(int(self.uniform() * span), span - 1)

    def normal(self) -> float:
        u1 = self.uniform()
        u2 = self.bits() * (2.0 ** -32)
        return math.sqrt(-2.0 * math.log(u1)) * math.cos(2.0 * math.pi * u2)


# ----------------------------------------------------------------------------
# Workload configurations
# ----------------------------------------------------------------------------

@dataclass(frozen=True)
class Workload:
    name: str
    T: int
    d_s: int
    d_t: int
    V: int
    tau: float
    dtype: str          # "f32" or "bf16"
    seed: int
    layout: str         # "tiny", "tiny_alt", "packed", "ragged"
    n_traj: int = 1
    traj_len: int = 512
    correlated_teacher: bool = False
    logit_std: float = 2.0
    description: str = ""


WORKLOADS: Dict[str, Workload] = {
    "tiny_fp32": Workload(
        "tiny_fp32", T=64, d_s=64, d_t=128, V=1000, tau=1.0, dtype="f32", seed=0, layout="tiny",
        description="T=64 in 2 turns, first 24 masked, 40 response tokens; d_s=64, d_t=128, V=1000"),
    "qwen3_0p6b": Workload(
        "qwen3_0p6b", T=4096, d_s=1024, d_t=4096, V=151936, tau=1.0, dtype="bf16", seed=1,
        layout="packed", n_traj=8,
        description="Qwen3-0.6B-shaped student head, 8 x 512 packed multi-turn tokens"),
    "qwen3_1p7b": Workload(
        "qwen3_1p7b", T=16384, d_s=2048, d_t=4096, V=151936, tau=1.0, dtype="bf16", seed=2,
        layout="packed", n_traj=32,
        description="Qwen3-1.7B-shaped student head, 32 x 512 packed multi-turn tokens"),
    "qwen3_4b": Workload(
        "qwen3_4b", T=32768, d_s=2560, d_t=4096, V=151936, tau=1.0, dtype="bf16", seed=3,
        layout="packed", n_traj=64, correlated_teacher=True,
        description="Qwen3-4B-shaped student head, 64 x 512 packed tokens, correlated teacher"),
    "ragged_multiturn": Workload(
        "ragged_multiturn", T=65536, d_s=2048, d_t=4096, V=151936, tau=0.7, dtype="bf16", seed=4,
        layout="ragged", n_traj=64,
        description="64 trajectories x up to 30 turns, lognormal think-then-act responses"),
}


def scaled(w: Workload, **changes) -> Workload:
    """A copy of a workload with some fields replaced (smaller parity cases)."""
    d = dict(w.__dict__)
    d.update(changes)
    return Workload(**d)


@dataclass
class Layout:
    mask: np.ndarray          # [T] uint8, 1 = supervised response token
    seg_id: np.ndarray        # [T] int32, response id, -1 outside responses
    n_responses: int
    spans: List[Tuple[str, int, int]] = field(default_factory=list)  # (kind, start, length)


def _tiny_layout(T: int, alt: bool) -> Layout:
    mask = np.zeros(T, np.uint8)
    seg = np.full(T, -1, np.int32)
    spans = []
    if not alt:
        # literal reading: 24 masked prompt/observation tokens, then 40 response tokens in 2 turns
        mask[24:64] = 1
        seg[24:44] = 0
        seg[44:64] = 1
        spans = [("obs", 0, 24), ("resp", 24, 20), ("resp", 44, 20)]
    else:
        # alternative reading: each turn is 12 observation tokens then 20 response tokens
        for t in range(2):
            o = 32 * t
            mask[o + 12:o + 32] = 1
            seg[o + 12:o + 32] = t
            spans += [("obs", o, 12), ("resp", o + 12, 20)]
    return Layout(mask, seg, 2, spans)


def _packed_layout(w: Workload) -> Layout:
    """T tokens in trajectories of traj_len tokens: observation spans U[20,60] (masked)
    alternate with response spans U[40,90] (supervised); ~5% of responses carry a
    20-token masked inserted span (thinking-budget continuation text)."""
    d = Draws(w.seed, STREAM_LAYOUT)
    T = w.T
    mask = np.zeros(T, np.uint8)
    seg = np.full(T, -1, np.int32)
    spans = []
    rid = 0
    for b in range((T + w.traj_len - 1) // w.traj_len):
        pos, end = b * w.traj_len, min(T, (b + 1) * w.traj_len)
        while pos < end:
            n_obs = min(d.randint(20, 60), end - pos)
            spans.append(("obs", pos, n_obs))
            pos += n_obs
            if pos >= end:
                break
            n_resp = min(d.randint(40, 90), end - pos)
            mask[pos:pos + n_resp] = 1
            seg[pos:pos + n_resp] = rid
            spans.append(("resp", pos, n_resp))
            if d.uniform() < 0.05 and n_resp > 24:
                ins = pos + d.randint(1, n_resp - 21)
                mask[ins:ins + 20] = 0
                spans.append(("inserted", ins, 20))
            rid += 1
            pos += n_resp
    return Layout(mask, seg, rid, spans)


def _ragged_layout(w: Workload) -> Layout:
    """64 trajectories x up to 30 turns, filled round-robin until T tokens.
    Turn: observation U[50,400] (masked; the first turn adds a U[100,300] masked
    task prompt), reasoning with lognormal length (median 300, sigma 0.6), then a
    U[10,20]-token action; the response is clipped at 2048 tokens. Reasoning that
    runs past the 1,920-token first stage gets a 26-token masked inserted span
    before the action (thinking-budget continuation, evaluation budgets)."""
    d = Draws(w.seed, STREAM_LAYOUT)
    trajs: List[List[Tuple[str, int, int]]] = [[] for _ in range(w.n_traj)]  # (kind, length, resp)
    total = 0
    rid = 0
    for turn in range(30):
        for b in range(w.n_traj):
            if total >= w.T:
                break
            parts = []
            if turn == 0:
                parts.append(("obs", d.randint(100, 300), -1))
            parts.append(("obs", d.randint(50, 400), -1))
            reasoning = int(round(300.0 * math.exp(0.6 * d.normal())))
            reasoning = max(1, reasoning)
            action = d.randint(10, 20)
            inserted = 0
            if reasoning > 1920:
                reasoning = 1920
                inserted = 26
            resp_total = min(reasoning + inserted + action, 2048)
            action = resp_total - reasoning - inserted
            parts.append(("resp", reasoning, rid))
            if inserted:
                parts.append(("inserted", inserted, rid))
            if action > 0:
                parts.append(("resp", action, rid))
            rid += 1
            trajs[b].extend(parts)
            total += sum(p[1] for p in parts)
        if total >= w.T:
            break
    mask = np.zeros(w.T, np.uint8)
    seg = np.full(w.T, -1, np.int32)
    spans = []
    pos = 0
    used = set()
    for b in range(w.n_traj):
        for kind, n, r in trajs[b]:
            if pos >= w.T:
                break
            n = min(n, w.T - pos)
            if kind != "obs":
                seg[pos:pos + n] = r
                used.add(r)
            if kind == "resp":
                mask[pos:pos + n] = 1
            spans.append((kind, pos, n))
            pos += n
    # responses are renumbered densely in order of appearance
    if used:
        order = {r: i for i, r in enumerate(sorted(used))}
        seg = np.array([order[s] if s >= 0 else -1 for s in seg], np.int32)
    return Layout(mask, seg, len(used), spans)


def layout(w: Workload) -> Layout:
    if w.layout == "tiny":
        return _tiny_layout(w.T, alt=False)
    if w.layout == "tiny_alt":
        return _tiny_layout(w.T, alt=True)
    if w.layout == "packed":
        return _packed_layout(w)
    if w.layout == "ragged":
        return _ragged_layout(w)
    raise ValueError(f"unknown layout {w.layout}")


def torch_dtype(w: Workload) -> torch.dtype:
    return torch.float32 if w.dtype == "f32" else torch.bfloat16


def hidden_and_heads(w: Workload, device="cpu") -> Dict[str, torch.Tensor]:
    """H_s [T,d_s], H_t [T,d_t] ~ N(0,1); W_s [V,d_s], W_t [V,d_t] ~ N(0, (std/sqrt(d))^2),
    so that logits have standard deviation ~ logit_std. With correlated_teacher the
    teacher reuses the student's features: H_t[:, :d_s] = H_s, W_t[:, :d_s] = 0.8 W_s,
    the rest fresh noise with std 1.2/sqrt(d_t - d_s), so z_t = 0.8 z_s + noise."""
    dt = torch_dtype(w)
    H_s = normal_tensor(w.seed, STREAM_H_S, (w.T, w.d_s), 1.0, dt, device)
    W_s = normal_tensor(w.seed, STREAM_W_S, (w.V, w.d_s), w.logit_std / math.sqrt(w.d_s), dt, device)
    if not w.correlated_teacher:
        H_t = normal_tensor(w.seed, STREAM_H_T, (w.T, w.d_t), 1.0, dt, device)
        W_t = normal_tensor(w.seed, STREAM_W_T, (w.V, w.d_t), w.logit_std / math.sqrt(w.d_t), dt, device)
    else:
        extra = w.d_t - w.d_s
        if extra <= 0:
            raise ValueError("correlated teacher needs d_t > d_s")
        H_t = torch.empty((w.T, w.d_t), dtype=dt, device=device)
        H_t[:, :w.d_s] = H_s
        H_t[:, w.d_s:] = normal_tensor(w.seed, STREAM_H_T_EXTRA, (w.T, extra), 1.0, dt, device)
        W_t = torch.empty((w.V, w.d_t), dtype=dt, device=device)
        W_t[:, :w.d_s] = (W_s.to(torch.float32) * 0.8).to(dt)
        W_t[:, w.d_s:] = normal_tensor(w.seed, STREAM_W_T_EXTRA, (w.V, extra), 1.2 / math.sqrt(extra),
                                       dt, device)
    return {"H_s": H_s, "H_t": H_t, "W_s": W_s, "W_t": W_t}


def uniform_weights(seed: int, T: int) -> np.ndarray:
    """Seeded upstream weights in [0.5, 1.5) for parity tests (float64)."""
    bits = uniform_bits(stream_key(seed, STREAM_G), 0, T, "cpu")
    return 0.5 + (bits.to(torch.float64) + 0.5).numpy() * (2.0 ** -32)


def token_ids(seed: int, T: int, V: int) -> np.ndarray:
    """Seeded sampled-token ids in [0, V) (int32)."""
    bits = uniform_bits(stream_key(seed, STREAM_TOKENS), 0, T, "cpu").numpy()
    return ((bits.astype(np.uint64) * np.uint64(V)) >> np.uint64(32)).astype(np.int32)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """A host copy of a bf16 tensor as uint16 bit patterns."""
    if t.dtype != torch.bfloat16:
        raise TypeError("expected bf16")
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def host_values(t: torch.Tensor) -> np.ndarray:
    """Host copy in the oracle's input convention: bf16 as uint16 bits, else float32."""
    if t.dtype == torch.bfloat16:
        return bf16_bits(t)
    return t.detach().contiguous().cpu().to(torch.float32).numpy()
