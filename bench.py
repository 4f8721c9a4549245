#!/usr/bin/env python3
"""Benchmark: fused OPD reverse-KL forward+backward on one GB300.

One step = one call of opd_kl_fwd_bwd (row compaction, gather, fused
student/teacher LM-head forward with online log-sum-exp, combine, fused
recompute emitting dz, dH_s and dW_s GEMMs, scatter) over one synthetic packed
batch of the Qwen3-1.7B-shaped workload (T = 16,384 tokens, d_s = 2048,
d_t = 4096, V = 151,936, bf16). Metric: supervised response tokens per second.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Inputs stay resident in HBM for `value`; `e2e` repeats the measurement through
the same C ABI with the per-step inputs copied from pinned host memory (the next
step's copy overlapping the current step) and the per-token KL copied back every
step. W_s + W_t (1.87 GB) exceed L2 (129 MB), so
every step streams the heads from HBM. `--impl reference` times the float64
CPU oracle on a bounded row sample of the same workload instead.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
import shutil
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2609_36608_gb300 import synth  # noqa: E402

METRIC = "response tokens/s and % bf16 tensor peak, fused OPD KL fwd+bwd (1 GB300)"
UNIT = "response tokens/s"
DEFAULT_WORKLOAD = "qwen3_1p7b"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNEL_SOURCES = {
    "fused_logits_fwd": ["paper_2609_36608_gb300/csrc/opd_fused.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
    "fused_logits_bwd": ["paper_2609_36608_gb300/csrc/opd_fused.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
    "head_logits_fwd": ["paper_2609_36608_gb300/csrc/opd_fused.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
    "head_logits_bwd": ["paper_2609_36608_gb300/csrc/opd_fused.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
    "gemm_dH": ["paper_2609_36608_gb300/csrc/opd_gemm.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
    "gemm_dW": ["paper_2609_36608_gb300/csrc/opd_gemm.cu", "paper_2609_36608_gb300/csrc/opd_device.cuh"],
}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def load_peaks():
    """The measured peaks (or the fallback) and, when recorded, the median SM clock of the
    sustained bf16 measurement (key "sustained_mhz")."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        out = {k: float(d[k]) for k in FALLBACK_PEAKS}
    except (OSError, KeyError, ValueError):
        return dict(FALLBACK_PEAKS), "fallback"
    try:
        out["sustained_mhz"] = float(d["clocks_under_load"]["sm_mhz_median"])
    except (KeyError, TypeError, ValueError):
        pass
    return out, "measured"


# --------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples (every 50 ms) of the benchmarked GPU while the timed region runs."""

    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, device_index: int):
        self.rows = []
        self.proc = None
        self.thread = None
        exe = shutil.which("nvidia-smi")
        if exe is None:
            return
        ident = None
        try:
            ident = "GPU-" + str(torch.cuda.get_device_properties(device_index).uuid)
        except Exception:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES", "")
            ident = vis.split(",")[device_index] if vis else str(device_index)
        self.cmd = [exe, "-i", ident, "--query-gpu=" + ",".join(self.FIELDS), "--format=csv,noheader,nounits",
                    "-lms", "50"]

    def start(self):
        if not hasattr(self, "cmd"):
            return
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) == len(self.FIELDS):
                self.rows.append(parts)

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=5)

    def mark(self) -> int:
        return len(self.rows)

    def summary(self, start: int = 0, end=None):
        """Median SM clock, maximum, throttle reasons and peak power of the samples [start, end)."""
        rows = self.rows[start:end]
        if not rows:
            return None
        sm = [float(r[0]) for r in rows if re.match(r"^[\d.]+$", r[0])]
        mx = [float(r[1]) for r in rows if re.match(r"^[\d.]+$", r[1])]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[4 + i].lower().startswith("active")})
        pw = [float(r[2]) for r in rows if re.match(r"^[\d.]+$", r[2])]
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "power_w_max": max(pw) if pw else None,
                "power_w_median": float(np.median(pw)) if pw else None}


def choose_peak(clocks, peaks, peak_src):
    """The bf16 denominator for a kernel timed inside the benchmark's step: the sustained
    figure when the kernel ran under the power limiter (sw_power_cap seen, or the median SM
    clock below 95% of its maximum) at a clock no more than 5% above the one the sustained
    figure was measured at; else the burst figure. Without a clock record the burst figure
    (the larger one) is used. Returns (peak, description)."""
    capped = bool(clocks) and (
        "sw_power_cap" in (clocks.get("reasons") or [])
        or (clocks.get("sm_mhz") and clocks.get("sm_max_mhz") and clocks["sm_mhz"] < 0.95 * clocks["sm_max_mhz"]))
    if capped and clocks.get("sm_mhz") and peaks.get("sustained_mhz"):
        capped = clocks["sm_mhz"] <= 1.05 * peaks["sustained_mhz"]
    if capped:
        return peaks["bf16_tflops_sustained"], f"bf16_tflops_sustained of {peak_src} (the step ran power-capped)"
    return peaks["bf16_tflops"], f"bf16_tflops (burst) of {peak_src} (the step ran at full clock)"


# ------------------------------------------------------------------ distributed

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world, backend):
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group(backend=backend)


def barrier(world):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(x: float, world: int, device) -> float:
    if world == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank_step: int, steps: int, world: int, max_ms: float) -> float:
    """Units all ranks processed per second, over the slowest rank's time (weak scaling)."""
    return units_per_rank_step * steps * world / (max_ms / 1000.0)


def sum_over_ranks(x: int, world: int, device) -> int:
    if world == 1:
        return int(x)
    t = torch.tensor([int(x)], dtype=torch.int64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.SUM)
    return int(t.item())


def workload_from_args(args):
    """The named workload; --trajectories N shrinks a packed workload to N trajectories of its
    length (the same shapes per row and the same layout generator: the small case of the same
    kernels that the ncu captures use)."""
    w = synth.WORKLOADS[args.workload]
    n = getattr(args, "trajectories", 0) or 0
    if n:
        if w.layout != "packed":
            raise SystemExit("--trajectories applies to the packed workloads only")
        w = synth.scaled(w, name=f"{w.name}_{n}traj", n_traj=n, T=n * w.traj_len)
    return w


def rank_workload(w, rank: int):
    """Each rank's own batch under data parallelism: rank 0 keeps the workload's seed (its
    batch is the single-GPU batch), rank k draws another packed batch of the same shape."""
    return w if rank == 0 else synth.scaled(w, seed=w.seed + 1000 * rank)


# -------------------------------------------------------------------- flops

def step_flops(w, R):
    executed = R * w.V * (8 * w.d_s + 4 * w.d_t)
    algorithmic = R * w.V * (6 * w.d_s + 2 * w.d_t)
    return executed, algorithmic


def kernel_flops(name, w, R):
    if name in ("fused_logits_fwd", "fused_logits_bwd"):
        return 2.0 * R * w.V * (w.d_s + w.d_t)
    if name in ("gemm_dH", "gemm_dW"):
        return 2.0 * R * w.V * w.d_s
    return None


def source_hash(name):
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES.get(name, []):
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def recorded_traffic(name, workload, step_path="kl"):
    """DRAM bytes per launch from the committed ncu summary, if the kernel source still matches
    (profiles/<kernel>_<workload>.txt for the KL step, <kernel>_<path>_<workload>.txt otherwise)."""
    # the loss step runs the reverse-KL step's kernels on the same shapes
    tag = workload if step_path in ("kl", "kl_seqmean") else f"{step_path}_{workload}"
    path = os.path.join(ROOT, "profiles", f"{name}_{tag}.txt")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m_b = re.search(r"^dram_bytes_per_launch:\s*([\d.eE+]+)", text, re.M)
    m_h = re.search(r"^source_sha256:\s*([0-9a-f]{64})", text, re.M)
    if not m_b or not m_h or m_h.group(1) != source_hash(name):
        return None
    return float(m_b.group(1))


# ---------------------------------------------------------------- CPU oracle

def oracle_rate(w, host, lay, g, rows, threads):
    import oracle
    oracle.build()
    t0 = time.perf_counter()
    oracle.opd_kl(host["H_s"], host["H_t"], host["W_s"], host["W_t"], lay.mask, g, w.tau, rows=rows,
                  want_dH=True, want_dW=True, n_threads=threads)
    dt = time.perf_counter() - t0
    return len(rows) / dt, dt


def host_inputs(x):
    return {k: synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")}


def sample_rows(mask, n, offset=0):
    sup = np.flatnonzero(mask)
    if len(sup) == 0:
        return sup
    idx = (np.arange(n) * max(1, len(sup) // n) + offset) % len(sup)
    return sup[np.unique(idx)]


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return 0
    w = workload_from_args(args)
    lay = synth.layout(w)
    gen_dev = "cuda" if torch.cuda.is_available() else "cpu"
    x = synth.hidden_and_heads(w, gen_dev)
    host = host_inputs(x)
    del x
    g = np.where(lay.mask != 0, synth.uniform_weights(w.seed, w.T), 0.0)
    threads = os.cpu_count() or 1
    rows_per_step = args.ref_rows
    import oracle
    oracle.build()
    tokens = synth.token_ids(w.seed, w.T, w.V)

    def one(rows):
        if args.path in ("kl", "kl_seqmean"):
            oracle_rate(w, host, lay, g, rows, threads)
        elif args.path == "score":
            oracle.score(host["H_t"], host["W_t"], tokens, w.tau, rows=rows, n_threads=threads)
        else:
            oracle.surrogate(host["H_s"], host["W_s"], tokens, np.full(w.T, -7.0), np.full(w.T, -7.0), lay.mask,
                             np.ones(w.T), w.tau, rows=rows, n_threads=threads)

    for i in range(args.warmup):
        one(sample_rows(lay.mask, rows_per_step, 7 * i))
    t0 = time.perf_counter()
    n = 0
    for i in range(args.steps):
        rows = sample_rows(lay.mask, rows_per_step, 13 * i + 1)
        one(rows)
        n += len(rows)
    dt = time.perf_counter() - t0
    value = n / dt
    what = {"kl": "logits, KL, dH_s rows and their dW_s contribution",
            "kl_seqmean": "logits, KL, dH_s rows and their dW_s contribution (seq-mean-token-mean weights)",
            "score": "teacher log-partition and token log-probabilities",
            "surrogate": "student logits, dual-clip loss, dH_s rows and their dW_s contribution"}[args.path]
    sample = (f"{rows_per_step} supervised rows of {w.name} per step (full V={w.V}, d_s={w.d_s}, d_t={w.d_t}): "
              f"{what} in float64")
    out = {"impl": "reference", "metric": PATH_METRICS[args.path], "value": value, "unit": UNIT, "n_gpus": world,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * dt / max(args.steps, 1),
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "config": {"workload": w.name, "T": w.T, "d_s": w.d_s, "d_t": w.d_t, "V": w.V,
                                           "temperature": w.tau},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)
    return 0


# ------------------------------------------------------------------ GPU arm

PATH_METRICS = {
    "kl": METRIC,
    "surrogate": "response tokens/s, sampled-token dual-clip surrogate loss step fwd+bwd (1 GB300)",
    "score": "response tokens/s, teacher token scoring fwd (1 GB300)",
    "kl_seqmean": "response tokens/s, fused OPD KL loss step (seq-mean-token-mean on the device) fwd+bwd (1 GB300)",
}


def path_setup(path, w, lay, x, dev, opd_kl, world=1, rank=0):
    """Per-step device inputs (the tensors the e2e leg copies from the host each step), the
    step function over them, the output read back each step, and the step's FLOPs."""
    R = int(lay.mask.sum())
    mask = torch.from_numpy(lay.mask).to(dev)
    weights = torch.from_numpy(opd_kl.opd_seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)).to(dev)
    dtype = opd_kl.OPD_DTYPE_BF16 if w.dtype == "bf16" else opd_kl.OPD_DTYPE_F32
    if path == "kl" and world > 1:
        # token-sharded data parallelism: this rank's batch, the paper's batch loss over every
        # rank's rows (response ids made global), dW_s and L summed over the ranks each step
        from paper_2609_36608_gb300 import data_parallel
        seg, n_ids = data_parallel.global_response_ids(torch.from_numpy(lay.seg_id).to(dev))
        sharded = data_parallel.ShardedSeqMeanKL(w.T, w.d_s, w.d_t, w.V, n_ids, w.tau, device=dev, dtype=dtype)
        dH, dW = torch.empty(w.T, w.d_s, device=dev), torch.empty(w.V, w.d_s, device=dev)
        inputs = {"H_s": x["H_s"], "H_t": x["H_t"], "mask": mask, "seg_id": seg}

        def step(i):
            sharded.step(i["H_s"], i["H_t"], x["W_s"], x["W_t"], i["mask"], i["seg_id"], dH, dW)
        step.outputs = {"kl": sharded.kl, "dH": dH}
        executed, algorithmic = step_flops(w, R)
        return inputs, step, sharded.loss, sharded.ws, executed, algorithmic
    if path == "kl":
        prob = opd_kl.make_problem(w.T, w.d_s, w.d_t, w.V, dtype, w.tau)
        ws = opd_kl.allocate_workspace(prob, dev)
        kl, stats = torch.empty(w.T, device=dev), torch.empty(w.T, 3, device=dev)
        dH, dW = torch.empty(w.T, w.d_s, device=dev), torch.empty(w.V, w.d_s, device=dev)
        inputs = {"H_s": x["H_s"], "H_t": x["H_t"], "mask": mask, "grad": weights}

        def step(i):
            opd_kl.opd_kl_fwd_bwd(prob, i["H_s"], i["H_t"], x["W_s"], x["W_t"], i["mask"], i["grad"], kl, stats, dH,
                                  dW, False, ws)
        step.outputs = {"kl": kl, "dH": dH}
        executed, algorithmic = step_flops(w, R)
        return inputs, step, kl, ws, executed, algorithmic
    if path == "kl_seqmean":
        # the whole loss step: weights from response ids on the device, L = sum_i w_i KL_i, gradients of L
        prob = opd_kl.make_problem(w.T, w.d_s, w.d_t, w.V, dtype, w.tau)
        n_ids = int(lay.seg_id.max()) + 1
        ws = opd_kl.allocate_seq_mean_workspace(prob, n_ids, dev)
        loss, kl, stats = torch.empty(1, device=dev), torch.empty(w.T, device=dev), torch.empty(w.T, 3, device=dev)
        dH, dW = torch.empty(w.T, w.d_s, device=dev), torch.empty(w.V, w.d_s, device=dev)
        inputs = {"H_s": x["H_s"], "H_t": x["H_t"], "mask": mask, "seg_id": torch.from_numpy(lay.seg_id).to(dev)}

        def step(i):
            opd_kl.opd_kl_seq_mean_fwd_bwd(prob, i["H_s"], i["H_t"], x["W_s"], x["W_t"], i["mask"], i["seg_id"],
                                           n_ids, 1e-8, loss, kl, stats, dH, dW, False, ws)
        step.outputs = {"kl": kl, "dH": dH}
        executed, algorithmic = step_flops(w, R)
        return inputs, step, loss, ws, executed, algorithmic
    tokens = torch.from_numpy(synth.token_ids(w.seed, w.T, w.V)).to(dev)
    if path == "score":
        prob = opd_kl.make_problem(w.T, w.d_t, w.d_t, w.V, dtype, w.tau)
        ws = opd_kl.allocate_workspace(prob, dev, forward_only=True)
        lse, logp = torch.empty(w.T, device=dev), torch.empty(w.T, device=dev)
        inputs = {"H_t": x["H_t"], "tokens": tokens, "mask": mask}

        def step(i):
            opd_kl.opd_score_tokens(prob, i["H_t"], x["W_t"], i["tokens"], i["mask"], lse, logp, ws)
        step.outputs = {"lse": lse, "logp": logp}
        fl = 2.0 * R * w.V * w.d_t
        return inputs, step, logp, ws, fl, fl
    # surrogate: synthetic teacher and behaviour log-probabilities (the teacher enters only there)
    g = torch.Generator(device="cpu").manual_seed(w.seed)
    logp_teacher = (torch.randn(w.T, generator=g) - 7.0).to(dev)
    logp_old = (logp_teacher.cpu() + 0.3 * torch.randn(w.T, generator=g)).to(dev)
    if world > 1:
        # token-sharded data parallelism of the surrogate loss step, as for the reverse KL above
        from paper_2609_36608_gb300 import data_parallel
        seg, n_ids = data_parallel.global_response_ids(torch.from_numpy(lay.seg_id).to(dev))
        sharded = data_parallel.ShardedSurrogate(w.T, w.d_s, w.V, n_ids, w.tau, device=dev)
        dH, dW = torch.empty(w.T, w.d_s, device=dev), torch.empty(w.V, w.d_s, device=dev)
        inputs = {"H_s": x["H_s"], "tokens": tokens, "logp_old": logp_old, "logp_teacher": logp_teacher,
                  "mask": mask, "seg_id": seg}

        def step(i):
            sharded.step(i["H_s"], x["W_s"], i["tokens"], i["logp_old"], i["logp_teacher"], i["mask"], i["seg_id"],
                         dH, dW)
        step.outputs = {"loss": sharded.loss_tok, "logp": sharded.logp, "dH": dH}
        return inputs, step, sharded.loss, sharded.ws, 8.0 * R * w.V * w.d_s, 6.0 * R * w.V * w.d_s
    prob = opd_kl.make_problem(w.T, w.d_s, w.d_s, w.V, dtype, w.tau)
    ws = opd_kl.allocate_workspace(prob, dev)
    loss, logp = torch.empty(w.T, device=dev), torch.empty(w.T, device=dev)
    dH, dW = torch.empty(w.T, w.d_s, device=dev), torch.empty(w.V, w.d_s, device=dev)
    n_ids = int(lay.seg_id.max()) + 1
    seq_ws = torch.empty(opd_kl.opd_seq_mean_token_mean_workspace_size(n_ids), dtype=torch.uint8, device=dev)
    dev_w = torch.empty(w.T, device=dev)
    total = torch.empty(1, device=dev)
    inputs = {"H_s": x["H_s"], "tokens": tokens, "logp_old": logp_old, "logp_teacher": logp_teacher, "mask": mask,
              "seg_id": torch.from_numpy(lay.seg_id).to(dev)}

    def step(i):
        # weights on the device, the surrogate forward+backward, then the batch loss L
        opd_kl.opd_seq_mean_token_mean_device(i["seg_id"], i["mask"], n_ids, 1e-8, None, dev_w, None, seq_ws)
        opd_kl.opd_surrogate_fwd_bwd(prob, i["H_s"], x["W_s"], i["tokens"], i["logp_old"], i["logp_teacher"],
                                     i["mask"], dev_w, loss, logp, dH, dW, False, ws)
        opd_kl.opd_seq_mean_token_mean_device(i["seg_id"], i["mask"], n_ids, 1e-8, loss, None, total, seq_ws)
    step.outputs = {"loss": loss, "logp": logp, "dH": dH}
    step.oracle_inputs = {"logp_old": logp_old, "logp_teacher": logp_teacher}
    return inputs, step, total, ws, 8.0 * R * w.V * w.d_s, 6.0 * R * w.V * w.d_s


def path_kernel_flops(path, name, w, R):
    if path in ("kl", "kl_seqmean"):
        return kernel_flops(name, w, R)
    d = w.d_t if path == "score" else w.d_s
    if name in ("head_logits_fwd", "head_logits_bwd"):
        return 2.0 * R * w.V * d
    if name in ("gemm_dH", "gemm_dW"):
        return 2.0 * R * w.V * w.d_s
    return None


def path_cpu_baseline(path, w, lay, x, args, step=None):
    """The oracle, as it stands, on a bounded row sample of the same workload: on every host
    core, and on one core for a smaller sample. With the step's GPU outputs, also the parity of
    those rows (the bench's own launch configuration against the oracle)."""
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    rows = sample_rows(lay.mask, args.cpu_rows, 3)
    if path in ("kl", "kl_seqmean"):
        host = host_inputs(x)
        g = np.where(lay.mask != 0, opd_seq_weights(lay), 0.0)

        def run(rs, n):
            return oracle.opd_kl(host["H_s"], host["H_t"], host["W_s"], host["W_t"], lay.mask, g, w.tau, rows=rs,
                                 want_dH=True, want_dW=True, n_threads=n)
        what = "float64 logits, KL, dH_s rows and their dW_s contribution"
    else:
        tokens = synth.token_ids(w.seed, w.T, w.V)
        if path == "score":
            H, W = synth.host_values(x["H_t"]), synth.host_values(x["W_t"])

            def run(rs, n):
                return oracle.score(H, W, tokens, w.tau, rows=rs, n_threads=n)
            what = "float64 teacher log-partition and token log-probabilities"
        else:
            # the GPU step's own behaviour and teacher log-probabilities and seq-mean weights
            H, W = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
            extra = getattr(step, "oracle_inputs", {})
            lo = extra["logp_old"].double().cpu().numpy() if extra else np.full(w.T, -7.0)
            lt = extra["logp_teacher"].double().cpu().numpy() if extra else np.full(w.T, -7.0)
            sw = opd_seq_weights(lay)

            def run(rs, n):
                return oracle.surrogate(H, W, tokens, lo, lt, lay.mask, sw, w.tau, rows=rs, n_threads=n)
            what = "float64 student logits, dual-clip loss, dH_s rows and their dW_s contribution"

    def timed(rs, n):
        t0 = time.perf_counter()
        res = run(rs, n)
        return time.perf_counter() - t0, res

    dt, ref = timed(rows, threads)
    rows1 = rows[:max(1, min(len(rows), args.cpu_rows_1t))]
    dt1, _ = timed(rows1, 1)
    out = {"value": len(rows) / dt, "unit": UNIT, "cores": threads, "kind": "oracle",
           "sample": f"{len(rows)} supervised rows of {w.name}: {what} ({dt:.1f} s)",
           "value_1_thread": len(rows1) / dt1,
           "sample_1_thread": f"the first {len(rows1)} of those rows on one core ({dt1:.1f} s)"}
    return out, sampled_parity(path, rows, ref, getattr(step, "outputs", None))


def sampled_parity(path, rows, ref, outputs):
    """Errors of the timed GPU step's outputs on the oracle's sampled rows, against the
    parity bounds (KL and per-token loss: 1e-4 + 2e-3 |x|; dH_s: 1e-2 relative Frobenius;
    lse and logp: 1e-4 + 1e-4 |x|)."""
    if not outputs:
        return None
    sel = torch.as_tensor(rows, device=next(iter(outputs.values())).device)
    pick = {k: v.index_select(0, sel).double().cpu().numpy() for k, v in outputs.items()}
    if path in ("kl", "kl_seqmean"):
        err = np.abs(pick["kl"] - ref.kl)
        rel = float(np.linalg.norm(pick["dH"] - ref.dH_s) / max(np.linalg.norm(ref.dH_s), 1e-300))
        return {"rows": len(rows), "kl_max_abs_err": float(err.max()),
                "kl_within_bound": bool((err <= 1e-4 + 2e-3 * np.abs(ref.kl)).all()),
                "dH_rel_fro_err": rel, "dH_within_bound": rel <= 1e-2}
    if path == "surrogate":
        e1, e2 = np.abs(pick["logp"] - ref.logp_s), np.abs(pick["loss"] - ref.loss)
        rel = float(np.linalg.norm(pick["dH"] - ref.dH_s) / max(np.linalg.norm(ref.dH_s), 1e-300))
        return {"rows": len(rows), "logp_max_abs_err": float(e1.max()), "loss_max_abs_err": float(e2.max()),
                "dH_rel_fro_err": rel,
                "within_bound": bool((e1 <= 1e-4 + 1e-4 * np.abs(ref.logp_s)).all()
                                     and (e2 <= 1e-4 + 2e-3 * np.abs(ref.loss)).all() and rel <= 1e-2)}
    if path == "score":
        lse_ref, lp_ref = ref
        e1, e2 = np.abs(pick["lse"] - lse_ref), np.abs(pick["logp"] - lp_ref)
        return {"rows": len(rows), "lse_max_abs_err": float(e1.max()), "logp_max_abs_err": float(e2.max()),
                "within_bound": bool((e1 <= 1e-4 + 1e-4 * np.abs(lse_ref)).all()
                                     and (e2 <= 1e-4 + 1e-4 * np.abs(lp_ref)).all())}
    return None


def opd_seq_weights(lay):
    import oracle
    return oracle.seq_mean_token_mean_weights(lay.seg_id, lay.mask)


def run_gpu(args):
    world, rank, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU (the reference arm runs with --impl reference)")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    init_dist(world, "nccl")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl

    w = rank_workload(workload_from_args(args), rank)
    lay = synth.layout(w)
    R = int(lay.mask.sum())
    R_job = sum_over_ranks(R, world, dev)  # supervised rows of all ranks' batches per step
    x = synth.hidden_and_heads(w, dev)
    inputs, step, result, ws, executed, algorithmic = path_setup(args.path, w, lay, x, dev, opd_kl, world, rank)

    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    for _ in range(args.warmup):
        step(inputs)
    torch.cuda.synchronize()
    if opd_kl.opd_kl_get_status(ws) != opd_kl.OPD_OK:
        raise RuntimeError("device status after warm-up is not OK")
    # Per-kernel times for the roofline come from K more steps with every library launch
    # bracketed by CUDA events on the launch stream: half of them just before the timed
    # region and half just after it, so that under the power limiter their clocks average out
    # to the timed region's. The timed region itself runs with the per-launch events off.
    prof = {}
    prof_ms = [0.0]
    prof_marks = []

    def kernel_pass(n):
        if n <= 0:
            return
        opd_kl.opd_kl_profile_start()
        q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        i0 = sampler.mark() if sampler else 0
        q0.record()
        for _ in range(n):
            step(inputs)
        q1.record()
        torch.cuda.synchronize()
        prof_marks.append((i0, sampler.mark() if sampler else 0))
        for name, (cnt, tot) in opd_kl.opd_kl_profile_stop().items():
            c0, t0 = prof.get(name, (0, 0.0))
            prof[name] = (c0 + cnt, t0 + tot)
        prof_ms[0] += q0.elapsed_time(q1)

    kernel_pass(args.steps // 2)
    barrier(world)
    torch.cuda.synchronize()
    mark0 = sampler.mark() if sampler else 0
    # the timed region: K steps, no per-launch events (the library's kernel timing is off)
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]  # end of each step
    ev0.record()
    for k in range(args.steps):
        step(inputs)
        marks[k].record()
    ev1.record()
    torch.cuda.synchronize()
    per_step = [ev0.elapsed_time(marks[0])] + [marks[k - 1].elapsed_time(marks[k]) for k in range(1, args.steps)]
    barrier(world)
    if opd_kl.opd_kl_get_status(ws) != opd_kl.OPD_OK:
        raise RuntimeError("device status after the timed region is not OK")
    ms = max_over_ranks(ev0.elapsed_time(ev1), world, dev)
    ms_step = ms / args.steps
    value = whole_job_rate(R_job, args.steps, 1, ms)
    clocks = sampler.summary(mark0, sampler.mark()) if sampler else None  # the timed region's samples

    kernel_pass(args.steps - args.steps // 2)
    ms_profiled = prof_ms[0] / args.steps
    if sampler:
        sampler.stop()
    clocks_kernel_pass = None
    if sampler and prof_marks:
        rows = [r for a, b in prof_marks for r in sampler.rows[a:b]]
        saved, sampler.rows = sampler.rows, rows
        clocks_kernel_pass = sampler.summary()
        sampler.rows = saved
    if opd_kl.opd_kl_get_status(ws) != opd_kl.OPD_OK:
        raise RuntimeError("device status after the per-kernel pass is not OK")

    # end to end through the same C ABI: every step's inputs come from pinned host memory
    # and its per-token result goes back to the host. Step i + 1's inputs are copied on a
    # second stream, into the other of two device buffers, while step i computes.
    host_in = {k: v.cpu().pin_memory() for k, v in inputs.items()}
    dev_in = [{k: torch.empty_like(v) for k, v in inputs.items()} for _ in range(2)]
    res_h = torch.empty(result.shape, dtype=result.dtype).pin_memory()
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = res_h.numel() * res_h.element_size()
    compute, copier = torch.cuda.current_stream(), torch.cuda.Stream()
    copied = [torch.cuda.Event(), torch.cuda.Event()]
    consumed = [torch.cuda.Event(), torch.cuda.Event()]

    def prefetch(b):
        with torch.cuda.stream(copier):
            copier.wait_event(consumed[b])  # the buffer's previous step has finished reading it
            for k, t in host_in.items():
                dev_in[b][k].copy_(t, non_blocking=True)
            copied[b].record(copier)

    def e2e_steps(n):
        for ev in consumed:  # copies of this run start after everything already on the compute stream
            ev.record(compute)
        prefetch(0)
        for i in range(n):
            b = i % 2
            if i + 1 < n:
                prefetch(1 - b)
            compute.wait_event(copied[b])
            step(dev_in[b])
            consumed[b].record(compute)
            res_h.copy_(result, non_blocking=True)
            compute.synchronize()
            float(res_h.view(-1)[0])

    e2e_steps(1)
    barrier(world)
    sampler_e2e = ClockSampler(local) if rank == 0 else None
    if sampler_e2e:
        sampler_e2e.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    e2e_steps(args.steps)
    e1.record()
    torch.cuda.synchronize()
    if sampler_e2e:
        sampler_e2e.stop()
    barrier(world)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    e2e_value = whole_job_rate(R_job, args.steps, 1, e2e_ms)

    if rank != 0:
        torch.distributed.destroy_process_group() if world > 1 else None
        return 0

    peaks, peak_src = load_peaks()
    kernels = {}
    total_k = sum(v[1] for v in prof.values()) or 1.0
    for name, (n, tot) in sorted(prof.items(), key=lambda kv: -kv[1][1]):
        kernels[name] = {"launches": n, "ms_per_launch": tot / max(n, 1), "share": tot / total_k}
    heavy = [k for k in kernels if path_kernel_flops(args.path, k, w, R) is not None]
    dom = max(heavy, key=lambda k: kernels[k]["ms_per_launch"] * kernels[k]["launches"]) if heavy else None
    roofline = None
    if dom:
        per_launch = path_kernel_flops(args.path, dom, w, R)
        achieved = per_launch / (kernels[dom]["ms_per_launch"] / 1000.0) / 1e12
        # the per-kernel times come from the kernel passes, so their clocks pick the peak
        peak, peak_desc = choose_peak(clocks_kernel_pass or clocks, peaks, peak_src)
        traffic = recorded_traffic(dom, w.name, args.path)
        roofline = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                    "frac": achieved / peak, "traffic": traffic, "peak_source": peak_desc,
                    "frac_of_burst": achieved / peaks["bf16_tflops"],
                    "frac_of_sustained": achieved / peaks["bf16_tflops_sustained"],
                    # the same kernel at its kernel-pass share of the timed region's step time
                    "frac_at_timed_step": achieved / peak * ms_profiled / ms_step,
                    # per clock: scaled to the clock the sustained peak was measured at (when both are known)
                    "frac_sustained_per_clock": (achieved / peaks["bf16_tflops_sustained"] * peaks["sustained_mhz"]
                                                 / clocks_kernel_pass["sm_mhz"])
                    if clocks_kernel_pass and clocks_kernel_pass.get("sm_mhz") and peaks.get("sustained_mhz")
                    else None,
                    "algorithmic_flops_per_launch": per_launch}

    cpu, parity = None, None
    if world == 1 and not args.no_cpu_baseline:
        cpu, parity = path_cpu_baseline(args.path, w, lay, x, args, step)

    out = {
        "metric": PATH_METRICS[args.path], "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step,
        "ms_per_step_median": float(np.median(per_step)), "ms_per_step_min_max": [min(per_step), max(per_step)],
        "ms_per_step_kernel_pass": ms_profiled, "clocks_kernel_pass": clocks_kernel_pass,
        "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic: seeded counter-based generator, packed multi-turn layout with masked observations "
                "and inserted tokens",
        "config": {"workload": w.name, "T": w.T, "R": R, "R_all_ranks": R_job, "d_s": w.d_s, "d_t": w.d_t, "V": w.V,
                   "temperature": w.tau,
                   "parallelism": (f"dp{world}: token-sharded, one {w.T}-token batch per GPU, dW_s and the "
                                   "loss all-reduced each step" if world > 1 and args.path in ("kl", "surrogate")
                                   else "replicas" if world > 1 else "single"),
                   "l2": "inputs larger than L2 (W_s + W_t = %.2f GB)" % ((w.d_s + w.d_t) * w.V * 2 / 1e9)},
        "tflops_executed": executed / (ms_step / 1000.0) / 1e12,
        "tflops_algorithmic": algorithmic / (ms_step / 1000.0) / 1e12,
        "pct_bf16_peak_executed": 100.0 * executed / (ms_step / 1000.0) / 1e12 / peaks["bf16_tflops"],
        "roofline": roofline,
        "cpu_baseline": cpu,
        "parity_sampled_rows": parity,
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "ms_per_step": e2e_ms / args.steps, "clocks": sampler_e2e.summary() if sampler_e2e else None},
        # launches in the timed region: the per-kernel pass runs the same K steps
        "gpu_launches": int(sum(v["launches"] for v in kernels.values())),
        "clocks": clocks,
        "kernels": kernels,
    }
    if args.path != "kl":
        out["path"] = args.path
    print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_calibration(args):
    """Sustained comparison under the board power cap: cuBLAS bf16 8192^3 (torch.matmul, a library
    reference point, not part of the step), then the fused step and the forward alone, each for
    args.calibrate seconds with clocks and power sampled every 50 ms. One JSON line per run."""
    if not torch.cuda.is_available():
        raise SystemExit("--calibrate needs a CUDA GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl

    def sustained(name, fn, flops):
        fn()
        torch.cuda.synchronize()
        sampler = ClockSampler(0)
        sampler.start()
        n, t0 = 0, time.time()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        while time.time() - t0 < args.calibrate:
            for _ in range(4):
                fn()
            n += 4
            torch.cuda.synchronize()
        e1.record()
        torch.cuda.synchronize()
        sampler.stop()
        ms = e0.elapsed_time(e1)
        print(json.dumps({"calibration": name, "calls": n, "ms_per_call": ms / n,
                          "tflops": flops * n / (ms / 1e3) / 1e12, "clocks": sampler.summary()}), flush=True)

    a = torch.randn(8192, 8192, device="cuda", dtype=torch.bfloat16)
    b = torch.randn(8192, 8192, device="cuda", dtype=torch.bfloat16)
    sustained("cublas_bf16_8192", lambda: torch.matmul(a, b), 2.0 * 8192 ** 3)
    del a, b
    w = workload_from_args(args)
    lay = synth.layout(w)
    R = int(lay.mask.sum())
    x = synth.hidden_and_heads(w, "cuda")
    prob = opd_kl.make_problem(w.T, w.d_s, w.d_t, w.V, opd_kl.OPD_DTYPE_BF16, w.tau)
    ws = opd_kl.allocate_workspace(prob)
    mask = torch.from_numpy(lay.mask).cuda()
    grad = torch.from_numpy(opd_kl.opd_seq_mean_token_mean_weights(lay.seg_id, lay.mask)).cuda()
    kl, st = torch.empty(w.T, device="cuda"), torch.empty(w.T, 3, device="cuda")
    dH, dW = torch.empty(w.T, w.d_s, device="cuda"), torch.empty(w.V, w.d_s, device="cuda")
    executed, _ = step_flops(w, R)
    sustained(f"fwd_bwd_{w.name}", lambda: opd_kl.opd_kl_fwd_bwd(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"],
                                                                 mask, grad, kl, st, dH, dW, False, ws), executed)
    sustained(f"fwd_{w.name}", lambda: opd_kl.opd_kl_forward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask,
                                                             kl, st, ws), 2.0 * R * w.V * (w.d_s + w.d_t))
    return 0


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--path", default="kl", choices=sorted(PATH_METRICS),
                    help="kl: the reverse-KL step (default, the headline); kl_seqmean: the same step "
                         "with the paper's batch loss aggregated on the device; surrogate: the "
                         "sampled-token dual-clip surrogate; score: teacher token scoring")
    ap.add_argument("--trajectories", type=int, default=0, metavar="N",
                    help="a packed workload cut to N trajectories (a small case for profiling)")
    ap.add_argument("--cpu-rows", type=int, default=48, help="row sample of the CPU-oracle baseline")
    ap.add_argument("--cpu-rows-1t", type=int, default=4, help="rows of the one-core CPU-oracle sample")
    ap.add_argument("--ref-rows", type=int, default=16, help="rows per step of --impl reference (the oracle splits rows over the host cores)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--calibrate", type=float, default=0.0, metavar="SECONDS",
                    help="instead of the benchmark: sustained cuBLAS vs fused-step runs under the power cap")
    args = ap.parse_args()
    if args.calibrate > 0:
        return run_calibration(args)
    if args.warmup < 3:
        log("note: at least 3 warm-up steps are required for a valid measurement; using 3")
        args.warmup = 3
    if args.impl == "reference":
        return run_reference(args)
    return run_gpu(args)


if __name__ == "__main__":
    sys.exit(main())
