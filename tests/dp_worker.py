"""One rank of the token-sharded data-parallel CPU test (torch.distributed.run, gloo).

The rank takes its contiguous rows of one small packed batch (row_shards), builds its
histogram of response ids (standing in for the device pass opd_seq_mean_token_mean_counts),
sums it over the ranks with the library's Reducer, computes its rows' KL, dH_s and dW_s part
with the float64 oracle under the whole batch's seq-mean-token-mean weights, and sums dW_s
(in several buckets) and its part of the loss over the ranks; then the same for the dual-clip
surrogate. The parent test compares the results with one oracle call over the whole batch."""

import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402
import torch.distributed as dist  # noqa: E402

import oracle  # noqa: E402
from paper_2609_36608_gb300 import data_parallel as dp  # noqa: E402
from paper_2609_36608_gb300 import synth  # noqa: E402


def batch():
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="dp_small", T=300, d_s=32, d_t=48, V=200, tau=0.8,
                     n_traj=3, traj_len=100, seed=5)
    return w, synth.layout(w)


def surrogate_inputs(w):
    """Sampled tokens and behaviour / teacher log-probabilities: the log-ratios spread over the
    ratio clip and the advantages take both signs."""
    rng = np.random.default_rng(7)
    tokens = synth.token_ids(w.seed, w.T, w.V)
    logp_teacher = rng.normal(-6.0, 1.0, w.T)
    logp_old = logp_teacher + rng.normal(0.0, 1.0, w.T)
    return tokens, logp_old, logp_teacher


def main():
    dist.init_process_group("gloo")
    world, rank = dist.get_world_size(), dist.get_rank()
    w, lay = batch()
    x = synth.hidden_and_heads(w, "cpu")
    host = [synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")]
    n_ids = int(lay.seg_id.max()) + 1
    lo, hi = dp.row_shards(w.T, world, lay.mask)[rank]
    counts = torch.zeros(2 * n_ids, dtype=torch.int32)
    for i in range(lo, hi):
        b = int(lay.seg_id[i])
        if b >= 0:
            counts[b] += int(lay.mask[i] != 0)
            counts[n_ids + b] += 1
    red = dp.Reducer(bucket_bytes=7 * w.d_s * 8)  # 7 vocabulary rows per bucket: 29 buckets
    red.sum_(counts)
    g = oracle.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
    rows = np.arange(lo, hi)
    res = oracle.opd_kl(*host, lay.mask, g, w.tau, rows=rows, want_dH=True, want_dW=True, n_threads=1)
    dW = torch.from_numpy(np.ascontiguousarray(res.dW_s))
    for work in red.sum_rows_(dW, async_op=True):
        work.wait()
    loss = torch.tensor([float(np.sum(g[rows] * res.kl))], dtype=torch.float64)
    red.sum_(loss)
    # the dual-clip surrogate under the same sharding (its per-token losses weighted alike)
    tokens, logp_old, logp_teacher = surrogate_inputs(w)
    sres = oracle.surrogate(host[0], host[2], tokens, logp_old, logp_teacher, lay.mask, g, w.tau, rows=rows,
                            n_threads=1)
    sdW = torch.from_numpy(np.ascontiguousarray(sres.dW_s))
    red.sum_rows_(sdW)
    sloss = torch.tensor([float(np.sum(g[rows] * sres.loss))], dtype=torch.float64)
    red.sum_(sloss)
    # global ids for batches packed per rank: rank k holds 3 + k local responses
    local = torch.tensor([-1, 0, 0, 1, -1, 2 + rank], dtype=torch.int32)
    gids, n_ids_all = dp.global_response_ids(local)
    np.savez(os.path.join(os.environ["OPD_TEST_OUT"], f"rank{rank}.npz"), lo=lo, hi=hi, counts=counts.numpy(),
             gids=gids.numpy(), n_ids_all=n_ids_all,
             kl=res.kl, dH=res.dH_s, dW=dW.numpy(), loss=loss.numpy(), buckets=len(red.buckets(w.V, w.d_s * 8)),
             s_loss_tok=sres.loss, s_dH=sres.dH_s, s_dW=sdW.numpy(), s_loss=sloss.numpy())
    dist.destroy_process_group()


if __name__ == "__main__":
    main()
