"""Token-sharded data parallelism of the OPD loss step, one process per GPU (torch.distributed).

The paper trains the student on two GPUs with a budget of 16,384 tokens per GPU (Appendix C,
training hyperparameters). Its loss over a batch B is the seq-mean-token-mean of per-token
losses (Appendix B.4, Eq. opd-surrogate), here of the per-token reverse KL (Section 3,
Eq. reverse-kl). Rows are independent for KL_i and dH_s[i, :], so the rows of a packed batch
split across processes with no exchange for those; two things need one:

  * the weights w_i = m_i / (|B| (n_b + eps)) count the supervised rows n_b of each response
    and the responses |B| of the whole batch: a sum over processes of a [2, n_ids] int32
    histogram (supervised rows and all rows per response id; 8 n_ids bytes);
  * dW_s = sum_i dz_i^T H_s[i, :] sums over every row of the batch: a sum over processes of
    the [V, d_s] fp32 gradient (1.24 GB at the Qwen3-1.7B shape), and of the scalar loss.

One step on every rank (device work in the library's kernels; this module only orders the
calls and the collectives, on each rank's own buffers):

  1. opd_seq_mean_token_mean_counts over the rank's rows;
  2. all-reduce (sum) of the histogram;
  3. opd_seq_mean_token_mean_from_counts: the rank's weights w;
  4. opd_kl_fwd_bwd with grad_kl = w: KL, stats, dH_s of the rank's rows, the rank's dW_s part;
  5. opd_seq_mean_token_mean_from_counts with loss_in = KL: the rank's part of L;
  6. all-reduce (sum) of dW_s, in buckets of whole vocabulary rows, and of L.

The result on every rank equals one call over the whole batch (up to the order of the dW_s
and L sums). A response may straddle two ranks: its rows' counts meet in step 2.

ShardedSeqMeanKL runs these steps for the reverse KL. ShardedSurrogate runs them for the
sampled-token dual-clip surrogate that the paper optimises (Appendix B.4), with
opd_surrogate_fwd_bwd as step 4 and the per-token surrogate losses in step 5.

The collectives are torch.distributed all-reduces (NCCL between GPUs, gloo on the CPU) on
buffers the rank owns; no kernel of the library reads another GPU's memory.
"""

from __future__ import annotations

from typing import List, Optional, Sequence, Tuple

import numpy as np
import torch
import torch.distributed as dist


def row_shards(T: int, world: int, mask: Optional[Sequence[int]] = None) -> List[Tuple[int, int]]:
    """Contiguous row ranges [lo, hi), one per rank, covering [0, T) in order.

    With a mask the cuts balance the supervised rows (the tensor-core work of the step is
    proportional to them): rank k's range ends at the first row where the running count of
    supervised rows reaches round((k + 1) R / world). Without one the rows are split evenly."""
    if world < 1 or T < 0:
        raise ValueError("world must be >= 1 and T >= 0")
    if mask is None:
        cuts = [(T * k) // world for k in range(world + 1)]
    else:
        m = np.asarray(mask).reshape(-1) != 0
        if m.shape[0] != T:
            raise ValueError("mask must have T entries")
        csum = np.cumsum(m)
        R = int(csum[-1]) if T else 0
        cuts = [0]
        for k in range(1, world):
            target = (k * R + world // 2) // world
            cut = int(np.searchsorted(csum, target, side="left")) + 1 if target > 0 else 0
            cuts.append(min(max(cut, cuts[-1]), T))
        cuts.append(T)
    return [(cuts[k], cuts[k + 1]) for k in range(world)]


def global_response_ids(seg_id: torch.Tensor, group=None):
    """Response ids made global across the ranks, for batches whose responses each live on one
    rank (every rank packs its own batch, as under the paper's per-GPU token budget).

    Rank k's ids b >= 0 become b + k n_max, with n_max the largest local id count over the
    ranks (ids < 0, rows outside every response, stay as they are). Returns the new ids (same
    device and dtype) and the global id count n_max * world. One all-reduce of one integer;
    with no process group (or one rank) the ids come back unchanged."""
    n_local = int(seg_id.max().item()) + 1 if seg_id.numel() else 0
    if not _active(group):
        return seg_id.clone(), max(n_local, 1)
    t = torch.tensor([n_local], dtype=torch.int64, device=seg_id.device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX, group=group)
    n_max = max(int(t.item()), 1)
    rank, world = dist.get_rank(group), dist.get_world_size(group)
    return torch.where(seg_id >= 0, seg_id + rank * n_max, seg_id), n_max * world


def _active(group) -> bool:
    return dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1


class Reducer:
    """The step's collectives: sums over the ranks of the process group, in place.

    dW_s is reduced in buckets of whole vocabulary rows (contiguous slices of the row-major
    [V, d_s] gradient) of about `bucket_bytes` each, issued back to back, so the transfer of one
    bucket overlaps the reduction of the next inside the collective library."""

    def __init__(self, group=None, bucket_bytes: int = 256 << 20):
        if bucket_bytes < 1:
            raise ValueError("bucket_bytes must be positive")
        self.group = group
        self.bucket_bytes = int(bucket_bytes)

    @property
    def active(self) -> bool:
        return _active(self.group)

    def sum_(self, t: torch.Tensor) -> None:
        if self.active:
            dist.all_reduce(t, op=dist.ReduceOp.SUM, group=self.group)

    def buckets(self, rows: int, row_bytes: int) -> List[Tuple[int, int]]:
        per = max(1, self.bucket_bytes // max(1, row_bytes))
        return [(v0, min(rows, v0 + per)) for v0 in range(0, rows, per)]

    def sum_rows_(self, t: torch.Tensor, async_op: bool = False):
        """Sum a [rows, ...] tensor over the ranks bucket by bucket; with async_op the works of
        the buckets are returned (wait on each before reading t)."""
        if not self.active or t.shape[0] == 0:
            return []
        if not t.is_contiguous():
            raise ValueError("the gradient must be contiguous")
        row_bytes = t[0].numel() * t.element_size()
        works = [dist.all_reduce(t[v0:v1], op=dist.ReduceOp.SUM, group=self.group, async_op=async_op)
                 for v0, v1 in self.buckets(t.shape[0], row_bytes)]
        return works if async_op else []


class _ShardedLoss:
    """What the sharded loss steps share: the workspaces of the seq-mean-token-mean passes, the
    histogram summed over the ranks, this rank's weights, and the sums of dW_s and of the loss."""

    def __init__(self, T: int, n_ids: int, eps: float, device, group, bucket_bytes: int):
        from . import opd_kl
        self.lib = opd_kl
        self.reducer = Reducer(group, bucket_bytes)
        self.n_ids, self.eps, self.T = int(n_ids), float(eps), int(T)
        dev = torch.device(device)
        self.device = dev
        self.seq_ws = torch.empty(opd_kl.opd_seq_mean_token_mean_workspace_size(self.n_ids), dtype=torch.uint8,
                                  device=dev)
        self.counts = torch.empty(2 * self.n_ids, dtype=torch.int32, device=dev)
        self.weights = torch.empty(T, dtype=torch.float32, device=dev)
        self.loss = torch.empty(1, dtype=torch.float32, device=dev)

    def _weights(self, seg_id, mask) -> None:
        """Steps 1-3: this rank's histogram, its sum over the ranks, this rank's weights."""
        self.lib.opd_seq_mean_token_mean_counts(seg_id, mask, self.n_ids, self.counts, self.seq_ws)
        self.reducer.sum_(self.counts)
        self.lib.opd_seq_mean_token_mean_from_counts(seg_id, mask, self.n_ids, self.counts, self.eps, None,
                                                     self.weights, None, self.seq_ws)

    def _finish(self, seg_id, mask, per_token_loss, dW_s, reduce_grad: bool, async_grad: bool):
        """Steps 5-6: this rank's part of L, then the sums of dW_s and L over the ranks."""
        self.lib.opd_seq_mean_token_mean_from_counts(seg_id, mask, self.n_ids, self.counts, self.eps,
                                                     per_token_loss, None, self.loss, self.seq_ws)
        works = self.reducer.sum_rows_(dW_s, async_op=async_grad) if reduce_grad else []
        self.reducer.sum_(self.loss)
        return works


class ShardedSeqMeanKL(_ShardedLoss):
    """The paper's batch loss over the per-token reverse KL and its gradients, for one rank's
    rows of a batch sharded by rows (see the module docstring for the steps).

    Construct once per shape on each rank; `step` then runs without host synchronisation.
    T is this rank's row count (its shard of the batch); d_s, d_t and V are the heads' sizes.
    `n_ids` is the number of global response ids of the whole batch (every rank passes the
    same value); seg_id holds global ids. The workspaces are allocated here, once, through
    PyTorch; the library itself allocates nothing."""

    def __init__(self, T: int, d_s: int, d_t: int, V: int, n_ids: int, temperature: float = 1.0,
                 eps: float = 1e-8, device="cuda", group=None, bucket_bytes: int = 256 << 20,
                 dtype: Optional[int] = None):
        super().__init__(T, n_ids, eps, device, group, bucket_bytes)
        opd_kl = self.lib
        dt = opd_kl.OPD_DTYPE_BF16 if dtype is None else dtype
        self.problem = opd_kl.make_problem(T, d_s, d_t, V, dt, temperature)
        self.ws = opd_kl.allocate_workspace(self.problem, self.device)
        self.kl = torch.empty(T, dtype=torch.float32, device=self.device)
        self.stats = torch.empty(T, 3, dtype=torch.float32, device=self.device)

    def step(self, H_s, H_t, W_s, W_t, mask, seg_id, dH_s, dW_s, accumulate_dW: bool = False,
             reduce_grad: bool = True, async_grad: bool = False):
        """Writes this rank's kl (self.kl), dH_s rows and, summed over every rank, dW_s and the
        batch loss (self.loss[0], the same on every rank). With async_grad the dW_s buckets are
        still in flight on return: their works are returned, and dW_s may be read only after
        each has been waited on.

        Gradient accumulation over micro-batches: the sum over the ranks covers the whole dW_s
        buffer, earlier contents included, so pass accumulate_dW=True with reduce_grad=False for
        every micro-batch but the last, and reduce_grad=True (the default) with the last."""
        self._weights(seg_id, mask)
        self.lib.opd_kl_fwd_bwd(self.problem, H_s, H_t, W_s, W_t, mask, self.weights, self.kl, self.stats, dH_s,
                                dW_s, accumulate_dW, self.ws)
        return self._finish(seg_id, mask, self.kl, dW_s, reduce_grad, async_grad)


class ShardedSurrogate(_ShardedLoss):
    """The sampled-token dual-clip surrogate the paper optimises (Appendix B.4, Eq.
    opd-token-advantage, opd-ratio, opd-dual-clip, opd-surrogate) under the same row sharding:
    the seq-mean-token-mean weights of the whole batch from the summed histogram, this rank's
    opd_surrogate_fwd_bwd with those weights, then the sums of dW_s and of L over the ranks.
    T is this rank's row count; d and V are the student head's sizes; `params` holds the
    surrogate's constants (None: the paper's delta = 0.2, kappa = 3, clip 20). The teacher
    enters only through logp_teacher, scored beforehand (opd_score_tokens)."""

    def __init__(self, T: int, d: int, V: int, n_ids: int, temperature: float = 1.0, eps: float = 1e-8,
                 device="cuda", group=None, bucket_bytes: int = 256 << 20, params=None):
        super().__init__(T, n_ids, eps, device, group, bucket_bytes)
        opd_kl = self.lib
        self.problem = opd_kl.make_problem(T, d, d, V, opd_kl.OPD_DTYPE_BF16, temperature)
        self.ws = opd_kl.allocate_workspace(self.problem, self.device)
        self.params = params
        self.loss_tok = torch.empty(T, dtype=torch.float32, device=self.device)
        self.logp = torch.empty(T, dtype=torch.float32, device=self.device)

    def step(self, H_s, W_s, tokens, logp_old, logp_teacher, mask, seg_id, dH_s, dW_s, accumulate_dW: bool = False,
             reduce_grad: bool = True, async_grad: bool = False):
        """Writes this rank's per-token losses (self.loss_tok) and log-probabilities (self.logp),
        its dH_s rows and, summed over every rank, dW_s and L (self.loss[0]). accumulate_dW,
        reduce_grad and async_grad as for ShardedSeqMeanKL.step."""
        self._weights(seg_id, mask)
        self.lib.opd_surrogate_fwd_bwd(self.problem, H_s, W_s, tokens, logp_old, logp_teacher, mask, self.weights,
                                       self.loss_tok, self.logp, dH_s, dW_s, accumulate_dW, self.ws,
                                       params=self.params)
        return self._finish(seg_id, mask, self.loss_tok, dW_s, reduce_grad, async_grad)
