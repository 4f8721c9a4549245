"""Token-sharded data parallelism (the paper trains the student on two GPUs, Appendix C) on
the CPU: the row partition, the collectives' bucketing, and two gloo ranks whose sharded steps
(the reverse KL and the dual-clip surrogate), computed with the float64 oracle, equal one oracle
call over the whole batch."""

import os
import socket
import subprocess
import sys

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import data_parallel as dp
from paper_2609_36608_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("world", [1, 2, 3, 8])
def test_row_shards_cover_the_batch_and_balance_supervised_rows(world):
    for name in ("tiny_fp32", "qwen3_0p6b", "ragged_multiturn"):
        lay = synth.layout(synth.WORKLOADS[name])
        T, R = lay.mask.shape[0], int((lay.mask != 0).sum())
        shards = dp.row_shards(T, world, lay.mask)
        assert len(shards) == world and shards[0][0] == 0 and shards[-1][1] == T
        assert all(shards[k][1] == shards[k + 1][0] for k in range(world - 1))
        per = [int((lay.mask[lo:hi] != 0).sum()) for lo, hi in shards]
        assert sum(per) == R
        assert max(per) - min(per) <= 1, per
    even = dp.row_shards(10, 3)
    assert even == [(0, 3), (3, 6), (6, 10)]
    assert dp.row_shards(0, 2, np.zeros(0)) == [(0, 0), (0, 0)]
    with pytest.raises(ValueError):
        dp.row_shards(5, 0)


def test_reducer_buckets_are_whole_rows_covering_the_gradient():
    r = dp.Reducer(bucket_bytes=256 << 20)
    V, row_bytes = 151936, 2048 * 4
    b = r.buckets(V, row_bytes)
    assert b[0][0] == 0 and b[-1][1] == V and all(b[k][1] == b[k + 1][0] for k in range(len(b) - 1))
    assert all((v1 - v0) * row_bytes <= 256 << 20 for v0, v1 in b) and len(b) == 5
    assert dp.Reducer(bucket_bytes=1).buckets(3, 100) == [(0, 1), (1, 2), (2, 3)]
    # without a process group (or with one rank) the reductions leave tensors untouched
    t = torch.arange(6.0).reshape(3, 2)
    assert r.sum_rows_(t) == [] and torch.equal(t, torch.arange(6.0).reshape(3, 2))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_equal_one_whole_batch_oracle_call(tmp_path, oracle_mod):
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "tests", "dp_worker.py")]
    env = dict(os.environ, OMP_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="", OPD_TEST_OUT=str(tmp_path))
    out = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT, env=env)
    assert out.returncode == 0, out.stderr[-3000:]
    r = [np.load(tmp_path / f"rank{k}.npz") for k in range(2)]
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    import dp_worker
    w, lay = dp_worker.batch()
    x = synth.hidden_and_heads(w, "cpu")
    host = [synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")]
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
    whole = oracle_mod.opd_kl(*host, lay.mask, g, w.tau, want_dH=True, want_dW=True)
    n_ids = int(lay.seg_id.max()) + 1
    # the shards meet at one row and a response straddles the cut
    assert int(r[0]["lo"]) == 0 and int(r[0]["hi"]) == int(r[1]["lo"]) and int(r[1]["hi"]) == w.T
    cut = int(r[0]["hi"])
    assert lay.seg_id[cut - 1] == lay.seg_id[cut] >= 0
    # every rank holds the whole batch's histogram after the sum
    sup = np.bincount(lay.seg_id[(lay.seg_id >= 0) & (lay.mask != 0)], minlength=n_ids)
    rows = np.bincount(lay.seg_id[lay.seg_id >= 0], minlength=n_ids)
    for k in range(2):
        np.testing.assert_array_equal(r[k]["counts"], np.concatenate([sup, rows]))
    # row-local outputs are exact; the sums over ranks agree to rounding
    np.testing.assert_array_equal(np.concatenate([r[0]["kl"], r[1]["kl"]]), whole.kl)
    np.testing.assert_array_equal(np.concatenate([r[0]["dH"], r[1]["dH"]]), whole.dH_s)
    for k in range(2):
        assert int(r[k]["buckets"]) > 1
        np.testing.assert_allclose(r[k]["dW"], whole.dW_s, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r[k]["loss"][0], float(np.sum(g * whole.kl)), rtol=1e-12)
    # global response ids: n_max = 4 (rank 1's ids reach 3), so rank k's ids shift by 4 k
    assert int(r[0]["n_ids_all"]) == 8 and int(r[1]["n_ids_all"]) == 8
    np.testing.assert_array_equal(r[0]["gids"], [-1, 0, 0, 1, -1, 2])
    np.testing.assert_array_equal(r[1]["gids"], [-1, 4, 4, 5, -1, 7])
    # the dual-clip surrogate under the same split
    tokens, logp_old, logp_teacher = dp_worker.surrogate_inputs(w)
    sw = oracle_mod.surrogate(host[0], host[2], tokens, logp_old, logp_teacher, lay.mask, g, w.tau)
    np.testing.assert_array_equal(np.concatenate([r[0]["s_loss_tok"], r[1]["s_loss_tok"]]), sw.loss)
    np.testing.assert_array_equal(np.concatenate([r[0]["s_dH"], r[1]["s_dH"]]), sw.dH_s)
    assert np.abs(sw.dH_s).max() > 0  # some tokens inside the clip carry a gradient
    for k in range(2):
        np.testing.assert_allclose(r[k]["s_dW"], sw.dW_s, rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(r[k]["s_loss"][0], float(np.sum(g * sw.loss)), rtol=1e-12)
