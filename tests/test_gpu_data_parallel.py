"""GPU side of token-sharded data parallelism, on one GPU: the rows of one batch are cut into
shards as row_shards cuts them across ranks, and each shard runs through the C ABI as its
rank would. The histogram sum that the all-reduce performs between ranks is done here by
adding the shards' count buffers; nothing waits on another shard's kernels.

Checked against the float64 oracle on the whole batch: the seq-mean-token-mean weights from
summed counts (Appendix B.4, Eq. opd-surrogate), the per-token KL, dH_s rows, dW_s summed
over the shards, and the batch loss."""

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import synth

pytestmark = pytest.mark.gpu

KL_ABS, KL_REL, GRAD_REL = 1e-4, 2e-3, 1e-2


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl
    return opd_kl


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


def _batch(**kw):
    base = dict(name="dp", T=900, d_s=192, d_t=256, V=1500, tau=0.8, n_traj=3, traj_len=300, seed=61)
    base.update(kw)
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], **base)
    return w, synth.layout(w)


@pytest.mark.parametrize("world", [1, 2, 3])
def test_weights_from_counts_summed_over_shards(lib, oracle_mod, world):
    from paper_2609_36608_gb300 import data_parallel as dp
    for w, lay in (_batch(), _batch(name="dp_ragged", T=4000, n_traj=8, traj_len=500, seed=62)):
        n_ids = int(lay.seg_id.max()) + 1
        seg = torch.from_numpy(lay.seg_id).cuda()
        mask = torch.from_numpy(lay.mask).cuda()
        shards = dp.row_shards(w.T, world, lay.mask)
        ws = [torch.empty(lib.opd_seq_mean_token_mean_workspace_size(n_ids), dtype=torch.uint8, device="cuda")
              for _ in shards]
        counts = [torch.full((2 * n_ids,), -7, dtype=torch.int32, device="cuda") for _ in shards]
        for (lo, hi), c, s in zip(shards, counts, ws):
            lib.opd_seq_mean_token_mean_counts(seg[lo:hi], mask[lo:hi], n_ids, c, s)
        total = sum(counts)  # what the all-reduce leaves on every rank
        sup = np.bincount(lay.seg_id[(lay.seg_id >= 0) & (lay.mask != 0)], minlength=n_ids)
        rows = np.bincount(lay.seg_id[lay.seg_id >= 0], minlength=n_ids)
        np.testing.assert_array_equal(total.cpu().numpy(), np.concatenate([sup, rows]))
        loss_in = torch.from_numpy(np.random.default_rng(world).random(w.T).astype(np.float32)).cuda()
        wt = torch.full((w.T,), float("nan"), device="cuda")
        parts = torch.zeros(len(shards), device="cuda")
        for k, ((lo, hi), s) in enumerate(zip(shards, ws)):
            lib.opd_seq_mean_token_mean_from_counts(seg[lo:hi], mask[lo:hi], n_ids, total, 1e-8, loss_in[lo:hi],
                                                    wt[lo:hi], parts[k:k + 1], s)
        torch.cuda.synchronize()
        for s in ws:
            assert lib.opd_kl_get_status(s) == lib.OPD_OK
        ref = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
        np.testing.assert_allclose(wt.cpu().numpy(), ref, rtol=2e-7, atol=0)
        want = float(np.sum(ref * loss_in.cpu().numpy().astype(np.float64)))
        assert abs(float(parts.sum()) - want) <= 1e-6 * abs(want)


def test_counts_report_an_id_beyond_n_ids(lib):
    seg = torch.tensor([0, 1, 5, -1], dtype=torch.int32, device="cuda")
    mask = torch.ones(4, dtype=torch.uint8, device="cuda")
    ws = torch.empty(lib.opd_seq_mean_token_mean_workspace_size(2), dtype=torch.uint8, device="cuda")
    c = torch.empty(4, dtype=torch.int32, device="cuda")
    lib.opd_seq_mean_token_mean_counts(seg, mask, 2, c, ws)
    w = torch.empty(4, device="cuda")
    lib.opd_seq_mean_token_mean_from_counts(seg, mask, 2, c, 1e-8, None, w, None, ws)
    assert lib.opd_kl_get_status(ws) == lib.OPD_ERR_INVALID_ARG  # the histogram pass's report survives
    assert c.cpu().tolist() == [1, 1, 1, 1]
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK


@pytest.mark.parametrize("world", [1, 2, 3])
def test_sharded_step_equals_the_whole_batch(lib, oracle_mod, world):
    """Each shard runs ShardedSeqMeanKL's calls (counts, summed counts, weights, fused step,
    its part of the loss); the shards' dW_s parts and losses are then summed as the all-reduce
    would sum them. With one shard this is ShardedSeqMeanKL.step itself."""
    from paper_2609_36608_gb300 import data_parallel as dp
    w, lay = _batch()
    x = synth.hidden_and_heads(w, "cuda")
    n_ids = int(lay.seg_id.max()) + 1
    seg = torch.from_numpy(lay.seg_id).cuda()
    mask = torch.from_numpy(lay.mask).cuda()
    shards = dp.row_shards(w.T, world, lay.mask)
    steps = [dp.ShardedSeqMeanKL(hi - lo, w.d_s, w.d_t, w.V, n_ids, w.tau) for lo, hi in shards]
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    dWs = [torch.full((w.V, w.d_s), float("nan"), device="cuda") for _ in shards]
    if world == 1:
        steps[0].step(x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, seg, dH, dWs[0])
        kl, loss, dW = steps[0].kl, steps[0].loss, dWs[0]
    else:
        counts = []
        for st, (lo, hi) in zip(steps, shards):
            lib.opd_seq_mean_token_mean_counts(seg[lo:hi], mask[lo:hi], n_ids, st.counts, st.seq_ws)
            counts.append(st.counts)
        total = sum(counts)
        kl = torch.empty(w.T, device="cuda")
        loss = torch.zeros(1, device="cuda")
        for st, (lo, hi), dW_k in zip(steps, shards, dWs):
            st.counts.copy_(total)
            args = (seg[lo:hi], mask[lo:hi], n_ids, st.counts, st.eps)
            lib.opd_seq_mean_token_mean_from_counts(*args, None, st.weights, None, st.seq_ws)
            lib.opd_kl_fwd_bwd(st.problem, x["H_s"][lo:hi], x["H_t"][lo:hi], x["W_s"], x["W_t"], mask[lo:hi],
                               st.weights, st.kl, st.stats, dH[lo:hi], dW_k, False, st.ws)
            lib.opd_seq_mean_token_mean_from_counts(*args, st.kl, None, st.loss, st.seq_ws)
            kl[lo:hi] = st.kl
            loss += st.loss
        dW = sum(dWs)
    torch.cuda.synchronize()
    for st in steps:
        assert lib.opd_kl_get_status(st.ws) == lib.OPD_OK and lib.opd_kl_get_status(st.seq_ws) == lib.OPD_OK
    host = [synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")]
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
    ref = oracle_mod.opd_kl(*host, lay.mask, g.astype(np.float32).astype(np.float64), w.tau)
    got = kl.cpu().numpy().astype(np.float64)
    assert (np.abs(got - ref.kl) <= KL_ABS + KL_REL * np.abs(ref.kl)).all()
    assert _rel(dH.cpu().numpy(), ref.dH_s) <= GRAD_REL
    assert _rel(dW.cpu().numpy(), ref.dW_s) <= GRAD_REL
    want = float(np.sum(g * ref.kl))
    assert abs(float(loss[0]) - want) <= 1e-4 * abs(want) + 1e-7


def test_bench_data_parallel_step_in_a_process_group_of_one(lib, oracle_mod, tmp_path):
    """bench.py's N > 1 step (path_setup with world > 1: global response ids, ShardedSeqMeanKL,
    the collectives) run as rank 0 of a one-rank NCCL process group: the collectives are then
    identities, and the loss and gradients must equal one whole-batch opd_kl_seq_mean_fwd_bwd call."""
    import torch.distributed as dist
    import bench
    from paper_2609_36608_gb300 import data_parallel as dp
    w, lay = _batch(name="dp_bench", T=1200, n_traj=4, seed=63)
    x = synth.hidden_and_heads(w, "cuda")
    dev = torch.device("cuda", torch.cuda.current_device())
    dist.init_process_group("nccl", init_method=f"file://{tmp_path}/pg", world_size=1, rank=0)
    try:
        inputs, step, result, ws, executed, algorithmic = bench.path_setup("kl", w, lay, x, dev, lib, world=2,
                                                                           rank=0)
        step(inputs)
        torch.cuda.synchronize()
        assert lib.opd_kl_get_status(ws) == lib.OPD_OK
        assert not dp.Reducer().active  # one rank: the sums over ranks leave every buffer as it is
        loss = float(result[0])
        kl = step.outputs["kl"].cpu().numpy()
        dH = step.outputs["dH"].cpu().numpy()
    finally:
        dist.destroy_process_group()
    n_ids = int(lay.seg_id.max()) + 1
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws2 = lib.allocate_seq_mean_workspace(prob, n_ids)
    loss2, kl2, st2 = torch.empty(1, device="cuda"), torch.empty(w.T, device="cuda"), torch.empty(w.T, 3, device="cuda")
    dH2, dW2 = torch.empty(w.T, w.d_s, device="cuda"), torch.empty(w.V, w.d_s, device="cuda")
    lib.opd_kl_seq_mean_fwd_bwd(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], torch.from_numpy(lay.mask).cuda(),
                                torch.from_numpy(lay.seg_id).cuda(), n_ids, 1e-8, loss2, kl2, st2, dH2, dW2, False,
                                ws2)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(kl, kl2.cpu().numpy())
    assert _rel(dH, dH2.cpu().numpy().astype(np.float64)) < 1e-5
    assert abs(loss - float(loss2[0])) <= 1e-6 * abs(float(loss2[0]))
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
    ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), lay.mask,
                            g.astype(np.float32).astype(np.float64), w.tau, want_dW=False)
    want = float(np.sum(g * ref.kl))
    assert abs(loss - want) <= 1e-4 * abs(want) + 1e-7


def test_shards_with_no_rows_and_loss_only_requests(lib, oracle_mod):
    """Degenerate shards: a rank whose row range is empty (T = 0) contributes a zero histogram and
    nothing else; a rank whose rows are all masked contributes only its responses' presence.
    from_counts with the loss alone (no weights buffer) gives that rank's part of L."""
    from paper_2609_36608_gb300 import data_parallel as dp
    w, lay = _batch(name="dp_edge", T=600, n_traj=2, seed=64)
    n_ids = int(lay.seg_id.max()) + 1
    seg = torch.from_numpy(lay.seg_id).cuda()
    mask = torch.from_numpy(lay.mask).cuda()
    # rank 0: nothing; rank 1: the first half with its mask cleared; rank 2: the rest
    half = w.T // 2
    shards = [(0, 0), (0, half), (half, w.T)]
    masks = [mask[0:0], torch.zeros(half, dtype=torch.uint8, device="cuda"), mask[half:]]
    eff_mask = np.concatenate([np.zeros(half, np.uint8), lay.mask[half:]])
    ws = [torch.empty(lib.opd_seq_mean_token_mean_workspace_size(n_ids), dtype=torch.uint8, device="cuda")
          for _ in shards]
    counts = [torch.full((2 * n_ids,), 5, dtype=torch.int32, device="cuda") for _ in shards]
    for (lo, hi), m, c, s in zip(shards, masks, counts, ws):
        lib.opd_seq_mean_token_mean_counts(seg[lo:hi], m, n_ids, c, s)
    assert (counts[0] == 0).all()
    total = sum(counts)
    loss_in = torch.from_numpy(np.random.default_rng(3).random(w.T).astype(np.float32)).cuda()
    parts = torch.full((3,), float("nan"), device="cuda")
    for k, ((lo, hi), m, s) in enumerate(zip(shards, masks, ws)):
        lib.opd_seq_mean_token_mean_from_counts(seg[lo:hi], m, n_ids, total, 1e-8, loss_in[lo:hi], None,
                                                parts[k:k + 1], s)
    torch.cuda.synchronize()
    for s in ws:
        assert lib.opd_kl_get_status(s) == lib.OPD_OK
    ref = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, eff_mask)
    p = parts.cpu().numpy().astype(np.float64)
    assert p[0] == 0.0 and p[1] == 0.0
    want = float(np.sum(ref * loss_in.cpu().numpy().astype(np.float64)))
    assert abs(p.sum() - want) <= 1e-6 * abs(want)
    assert dp.row_shards(w.T, 3, np.zeros(w.T, np.uint8)) == [(0, 0), (0, 0), (0, w.T)]


def _off_kinks(seed, n):
    """Log-ratio offsets in [-0.6, 1.4] at least 0.02 from the ratio clip's kinks (ln 0.8, ln 1.2)
    and the dual clip's (ln 3), so that fp32 and fp64 take the same branch."""
    edges = np.log([0.8, 1.2, 3.0])
    rng = np.random.default_rng(seed)
    out = rng.uniform(-0.6, 1.4, 4 * n)
    out = out[np.min(np.abs(out[:, None] - edges[None, :]), axis=1) > 0.02]
    return out[:n]


@pytest.mark.parametrize("world", [1, 2, 3])
def test_sharded_surrogate_equals_the_whole_batch(lib, oracle_mod, world):
    """ShardedSurrogate's calls per shard (with one shard: its step itself); the shards' dW_s
    parts and losses summed as the all-reduce sums them, against the float64 oracle's surrogate
    over the whole batch under the whole batch's seq-mean-token-mean weights."""
    from paper_2609_36608_gb300 import data_parallel as dp
    w, lay = _batch(name="dp_sur", T=900, d_s=160, V=1300, n_traj=3, seed=65)
    x = synth.hidden_and_heads(w, "cuda")
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    tokens = synth.token_ids(w.seed, w.T, w.V)
    _, lp_ref = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = (lp_ref - _off_kinks(world, w.T)).astype(np.float32)
    adv = np.random.default_rng(9).choice([-1.0, 1.0], w.T) * np.random.default_rng(10).uniform(0.2, 1.5, w.T)
    logp_teacher = (logp_old.astype(np.float64) + adv).astype(np.float32)
    n_ids = int(lay.seg_id.max()) + 1
    f32 = lambda a: torch.from_numpy(np.asarray(a, np.float32)).cuda()
    seg, mask = torch.from_numpy(lay.seg_id).cuda(), torch.from_numpy(lay.mask).cuda()
    tok, lo_t, lt_t = torch.from_numpy(tokens).cuda(), f32(logp_old), f32(logp_teacher)
    shards = dp.row_shards(w.T, world, lay.mask)
    steps = [dp.ShardedSurrogate(hi - lo, w.d_s, w.V, n_ids, w.tau) for lo, hi in shards]
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    dWs = [torch.full((w.V, w.d_s), float("nan"), device="cuda") for _ in shards]
    loss_tok = torch.empty(w.T, device="cuda")
    if world == 1:
        steps[0].step(x["H_s"], x["W_s"], tok, lo_t, lt_t, mask, seg, dH, dWs[0])
        loss, dW = steps[0].loss, dWs[0]
        loss_tok.copy_(steps[0].loss_tok)
    else:
        for st, (lo, hi) in zip(steps, shards):
            lib.opd_seq_mean_token_mean_counts(seg[lo:hi], mask[lo:hi], n_ids, st.counts, st.seq_ws)
        total = sum(st.counts for st in steps)
        loss = torch.zeros(1, device="cuda")
        for st, (lo, hi), dW_k in zip(steps, shards, dWs):
            st.counts.copy_(total)
            args = (seg[lo:hi], mask[lo:hi], n_ids, st.counts, st.eps)
            lib.opd_seq_mean_token_mean_from_counts(*args, None, st.weights, None, st.seq_ws)
            lib.opd_surrogate_fwd_bwd(st.problem, x["H_s"][lo:hi], x["W_s"], tok[lo:hi], lo_t[lo:hi], lt_t[lo:hi],
                                      mask[lo:hi], st.weights, st.loss_tok, st.logp, dH[lo:hi], dW_k, False, st.ws)
            lib.opd_seq_mean_token_mean_from_counts(*args, st.loss_tok, None, st.loss, st.seq_ws)
            loss_tok[lo:hi] = st.loss_tok
            loss += st.loss
        dW = sum(dWs)
    torch.cuda.synchronize()
    for st in steps:
        assert lib.opd_kl_get_status(st.ws) == lib.OPD_OK and lib.opd_kl_get_status(st.seq_ws) == lib.OPD_OK
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               lay.mask, g.astype(np.float32).astype(np.float64), w.tau)
    got = loss_tok.cpu().numpy().astype(np.float64)
    assert (np.abs(got - ref.loss) <= 1e-4 + 2e-3 * np.abs(ref.loss)).all()
    assert _rel(dH.cpu().numpy(), ref.dH_s) <= GRAD_REL
    assert _rel(dW.cpu().numpy(), ref.dW_s) <= GRAD_REL
    want = float(np.sum(g * ref.loss))
    assert abs(float(loss[0]) - want) <= 1e-4 * abs(want) + 1e-7


def test_bench_data_parallel_surrogate_step_in_a_process_group_of_one(lib, tmp_path):
    """bench.py's N > 1 surrogate step (ShardedSurrogate with global response ids) as rank 0 of
    a one-rank NCCL group equals the single-GPU surrogate loss step of the same batch."""
    import torch.distributed as dist
    import bench
    w, lay = _batch(name="dp_bench_sur", T=1200, n_traj=4, seed=66)
    x = synth.hidden_and_heads(w, "cuda")
    dev = torch.device("cuda", torch.cuda.current_device())
    dist.init_process_group("nccl", init_method=f"file://{tmp_path}/pg", world_size=1, rank=0)
    try:
        inputs, step, result, ws, _, _ = bench.path_setup("surrogate", w, lay, x, dev, lib, world=2, rank=0)
        step(inputs)
        torch.cuda.synchronize()
        assert lib.opd_kl_get_status(ws) == lib.OPD_OK
        dp_loss = float(result[0])
        dp_tok = step.outputs["loss"].cpu().numpy()
        dp_dH = step.outputs["dH"].cpu().numpy()
    finally:
        dist.destroy_process_group()
    inputs1, step1, result1, ws1, _, _ = bench.path_setup("surrogate", w, lay, x, dev, lib)
    step1(inputs1)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws1) == lib.OPD_OK
    np.testing.assert_array_equal(dp_tok, step1.outputs["loss"].cpu().numpy())
    assert _rel(dp_dH, step1.outputs["dH"].cpu().numpy().astype(np.float64)) < 1e-5
    ref = float(result1[0])
    assert abs(dp_loss - ref) <= 1e-6 * abs(ref) + 1e-9


def _random_dp_cases(n, seed=977):
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        T = int(rng.integers(1, 700))
        out.append(dict(T=T, d_s=8 * int(rng.integers(1, 33)), d_t=8 * int(rng.integers(1, 49)),
                        V=int(rng.integers(2, 3000)), tau=float(rng.choice([0.5, 1.0, 1.6])),
                        world=int(rng.integers(2, 6)), density=float(rng.uniform(0.0, 1.0)),
                        n_resp=int(rng.integers(1, 12)), seed=300 + i))
    return out


@pytest.mark.parametrize("case", _random_dp_cases(6), ids=lambda c: f"T{c['T']}-w{c['world']}-V{c['V']}")
def test_sharded_kl_random_shapes(lib, oracle_mod, case):
    """Seeded random problems split over 2-5 emulated ranks: random masks (density 0-1, so some
    shards may hold no supervised row) and random response layouts (responses straddle cuts). The
    summed dW_s and loss and the per-row KL and dH_s match the whole-batch oracle."""
    from paper_2609_36608_gb300 import data_parallel as dp
    rng = np.random.default_rng(case["seed"])
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="dp_rand", T=case["T"], d_s=case["d_s"], d_t=case["d_t"],
                     V=case["V"], tau=case["tau"], n_traj=1, traj_len=case["T"], seed=case["seed"])
    mask = (rng.random(w.T) < case["density"]).astype(np.uint8)
    seg = np.sort(rng.integers(-1, case["n_resp"], w.T)).astype(np.int32)
    n_ids = case["n_resp"]
    x = synth.hidden_and_heads(w, "cuda")
    seg_t, mask_t = torch.from_numpy(seg).cuda(), torch.from_numpy(mask).cuda()
    shards = dp.row_shards(w.T, case["world"], mask)
    steps = [dp.ShardedSeqMeanKL(hi - lo, w.d_s, w.d_t, w.V, n_ids, w.tau) for lo, hi in shards]
    for st, (lo, hi) in zip(steps, shards):
        lib.opd_seq_mean_token_mean_counts(seg_t[lo:hi], mask_t[lo:hi], n_ids, st.counts, st.seq_ws)
    total = sum(st.counts for st in steps)
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    kl = torch.empty(w.T, device="cuda")
    dW = torch.zeros(w.V, w.d_s, device="cuda")
    loss = torch.zeros(1, device="cuda")
    for st, (lo, hi) in zip(steps, shards):
        st.counts.copy_(total)
        args = (seg_t[lo:hi], mask_t[lo:hi], n_ids, st.counts, st.eps)
        lib.opd_seq_mean_token_mean_from_counts(*args, None, st.weights, None, st.seq_ws)
        dW_k = torch.empty(w.V, w.d_s, device="cuda")
        lib.opd_kl_fwd_bwd(st.problem, x["H_s"][lo:hi], x["H_t"][lo:hi], x["W_s"], x["W_t"], mask_t[lo:hi],
                           st.weights, st.kl, st.stats, dH[lo:hi], dW_k, False, st.ws)
        lib.opd_seq_mean_token_mean_from_counts(*args, st.kl, None, st.loss, st.seq_ws)
        kl[lo:hi] = st.kl
        dW += dW_k
        loss += st.loss
    torch.cuda.synchronize()
    for st in steps:
        assert lib.opd_kl_get_status(st.ws) == lib.OPD_OK and lib.opd_kl_get_status(st.seq_ws) == lib.OPD_OK
    g = oracle_mod.seq_mean_token_mean_weights(seg, mask)
    ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), mask,
                            g.astype(np.float32).astype(np.float64), w.tau)
    got = kl.cpu().numpy().astype(np.float64)
    assert (np.abs(got - ref.kl) <= KL_ABS + KL_REL * np.abs(ref.kl)).all()
    sup = mask != 0
    assert (dH.cpu().numpy()[~sup] == 0).all()
    if sup.any():
        assert _rel(dH.cpu().numpy(), ref.dH_s) <= GRAD_REL
        assert _rel(dW.cpu().numpy(), ref.dW_s) <= GRAD_REL
    else:
        assert (dW == 0).all()
    want = float(np.sum(g * ref.kl))
    assert abs(float(loss[0]) - want) <= 1e-4 * abs(want) + 1e-7
