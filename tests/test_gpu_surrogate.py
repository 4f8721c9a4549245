"""GPU parity of token scoring and the sampled-token surrogate (Appendix B.4) against
the float64 oracle, through the C ABI.

Tolerances: log-partition and log-probability |gpu - oracle| <= 1e-4 + 1e-4 |oracle|;
per-token surrogate loss |gpu - oracle| <= 1e-4 + 2e-3 |oracle|; dH_s and dW_s within
1e-2 relative Frobenius error (bf16 inputs, fp32 accumulation, bf16 dz).

The surrogate's gradient is piecewise (ratio clip, dual clip, log-ratio clip), so a
branch decision taken in fp32 on the GPU and in fp64 in the oracle could differ for a
token sitting on a kink. The small cases therefore build the behaviour-policy
log-probabilities from the oracle's own scores, keeping every token's log-ratio at least
0.02 away from ln 0.8, ln 1.2 and ln 3 (the GPU's log-probabilities differ from the
oracle's by ~1e-5).
"""

import math

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import synth

pytestmark = pytest.mark.gpu

EDGES = np.log([0.8, 1.2, 3.0])


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl
    return opd_kl


@pytest.fixture(params=["bn256/cta1", "pair256/pair"])
def tiling(request, monkeypatch):
    """Single-CTA and CTA-pair tilings of the head kernels and of the gradient GEMMs."""
    fused, gemm = request.param.split("/")
    monkeypatch.setenv("OPD_KL_FUSED", fused)
    monkeypatch.setenv("OPD_KL_GEMM", gemm)
    return request.param


def _case(**kw):
    base = dict(name="head", T=700, d_s=256, d_t=384, V=1000, tau=0.7, n_traj=7, traj_len=100, seed=31)
    base.update(kw)
    return synth.scaled(synth.WORKLOADS["qwen3_1p7b"], **base)


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


def _close(got, want, abs_tol, rel_tol, what):
    excess = np.abs(np.asarray(got, np.float64) - want) - (abs_tol + rel_tol * np.abs(want))
    assert excess.max() <= 0, f"{what}: worst excess {excess.max():.3e} at {int(excess.argmax())}"


def _score(lib, w, H, W, tokens, mask):
    prob = lib.make_problem(w.T, H.shape[1], H.shape[1], w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    lse = torch.full((w.T,), float("nan"), device="cuda")
    lp = torch.full((w.T,), float("nan"), device="cuda")
    lib.opd_score_tokens(prob, H, W, torch.from_numpy(tokens).cuda(), torch.from_numpy(mask).cuda(), lse, lp, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    return lse.cpu().numpy(), lp.cpu().numpy()


def _surrogate(lib, w, x, tokens, logp_old, logp_teacher, mask, weights, accumulate=False, dW_init=None):
    prob = lib.make_problem(w.T, w.d_s, w.d_s, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    f32 = lambda a: torch.from_numpy(np.asarray(a, np.float32)).cuda()
    loss = torch.full((w.T,), float("nan"), device="cuda")
    lp = torch.full((w.T,), float("nan"), device="cuda")
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    dW = torch.full((w.V, w.d_s), float("nan"), device="cuda") if dW_init is None else dW_init.clone()
    lib.opd_surrogate_fwd_bwd(prob, x["H_s"], x["W_s"], torch.from_numpy(tokens).cuda(), f32(logp_old),
                              f32(logp_teacher), torch.from_numpy(mask).cuda(), f32(weights), loss, lp, dH, dW,
                              accumulate, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    return loss.cpu().numpy(), lp.cpu().numpy(), dH.cpu().numpy(), dW.cpu().numpy()


def _clear_offsets(seed, n):
    rng = np.random.default_rng(seed)
    out = np.empty(n)
    for i in range(n):
        while True:
            r = rng.uniform(-0.6, 1.4)
            if np.min(np.abs(r - EDGES)) > 0.02:
                out[i] = r
                break
    return out


def test_score_tokens_small(lib, oracle_mod, tiling):
    w = _case()
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    for H, W in ((x["H_s"], x["W_s"]), (x["H_t"], x["W_t"])):
        lse, lp = _score(lib, w, H, W, tokens, lay.mask)
        sup = lay.mask != 0
        ref_lse, ref_lp = oracle_mod.score(synth.host_values(H), synth.host_values(W), tokens, w.tau,
                                           rows=np.flatnonzero(sup))
        _close(lse[sup], ref_lse, 1e-4, 1e-4, "lse")
        _close(lp[sup], ref_lp, 1e-4, 1e-4, "logp")
        assert (lse[~sup] == 0).all() and (lp[~sup] == 0).all()


def test_surrogate_small(lib, oracle_mod, tiling):
    w = _case(T=600, d_s=192, V=1237, tau=0.9, n_traj=6, seed=32)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    _, lp_ref = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = (lp_ref - _clear_offsets(1, w.T)).astype(np.float32)
    adv = np.random.default_rng(2).choice([-1.0, 1.0], w.T) * np.random.default_rng(3).uniform(0.2, 1.5, w.T)
    logp_teacher = (logp_old.astype(np.float64) + adv).astype(np.float32)
    weights = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask).astype(np.float32)
    loss, lp, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, lay.mask, weights)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               lay.mask, weights.astype(np.float64), w.tau)
    sup = lay.mask != 0
    _close(lp[sup], ref.logp_s[sup], 1e-4, 1e-4, "logp")
    _close(loss, ref.loss, 1e-4, 2e-3, "loss")
    assert (loss[~sup] == 0).all() and (dH[~sup] == 0).all()
    assert _rel(dH, ref.dH_s) <= 1e-2, _rel(dH, ref.dH_s)
    assert _rel(dW, ref.dW_s) <= 1e-2, _rel(dW, ref.dW_s)


@pytest.mark.parametrize("shape", [dict(T=50, d_s=8, V=2), dict(T=90, d_s=16, V=64)])
def test_surrogate_and_scoring_below_one_tile(lib, oracle_mod, shape, tiling):
    w = _case(n_traj=1, traj_len=shape["T"], seed=33, **shape)
    mask = (np.arange(w.T) % 4 != 2).astype(np.uint8)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    lse, lp = _score(lib, w, x["H_s"], x["W_s"], tokens, mask)
    sup = mask != 0
    ref_lse, ref_lp = oracle_mod.score(Hs, Ws, tokens, w.tau, rows=np.flatnonzero(sup))
    _close(lse[sup], ref_lse, 1e-4, 1e-4, "lse")
    _close(lp[sup], ref_lp, 1e-4, 1e-4, "logp")
    _, lp_full = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = (lp_full - _clear_offsets(4, w.T)).astype(np.float32)
    adv = np.random.default_rng(5).choice([-1.0, 1.0], w.T) * np.random.default_rng(6).uniform(0.2, 1.5, w.T)
    logp_teacher = (logp_old.astype(np.float64) + adv).astype(np.float32)
    weights = np.where(sup, 1.0 / max(int(sup.sum()), 1), 0.0).astype(np.float32)
    loss, lp2, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, mask, weights)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               mask, weights.astype(np.float64), w.tau)
    _close(loss, ref.loss, 1e-4, 2e-3, "loss")
    assert _rel(dH, ref.dH_s) <= 1e-2, _rel(dH, ref.dH_s)
    assert _rel(dW, ref.dW_s) <= 1e-2, _rel(dW, ref.dW_s)


def test_surrogate_log_ratio_clip_branch(lib, oracle_mod, tiling):
    """Tokens whose log-ratio r = logp - logp_old lies beyond the +-20 clip (Appendix B.4,
    Eq. opd-ratio), with both signs of the advantage, beside unclipped tokens.

    Five classes of supervised token, by row: r in [20.5, 40], r in [-40, -20.5], r in
    [100, 200] (exp(r) overflows fp32 unless r is clipped first), r in [-200, -100], and
    r in [-0.6, 1.4] off the ratio-clip kinks. Every r keeps at least 0.5 from +-20, far
    beyond the ~1e-5 difference between the GPU's and the oracle's log-probabilities, so
    both sides take the same branch. Beyond the clip the ratio is constant, so those
    tokens must carry no gradient at all: their dH_s rows are exactly zero. With A < 0 and
    r > 20 the dual clip caps the loss at -kappa A; with A < 0 and r < -20 the loss is
    -(1 - delta) A. A second call with every supervised token beyond the clip must give
    dH_s = 0 and dW_s = 0 exactly (a slope kept at r < -20 would leave ~1e-9 there)."""
    w = _case(T=600, d_s=192, V=1237, tau=0.9, n_traj=6, seed=35)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    _, lp_ref = oracle_mod.score(Hs, Ws, tokens, w.tau)
    rng = np.random.default_rng(35)
    cls = np.arange(w.T) % 5
    r = np.select([cls == 0, cls == 1, cls == 2, cls == 3],
                  [rng.uniform(20.5, 40, w.T), -rng.uniform(20.5, 40, w.T), rng.uniform(100, 200, w.T),
                   -rng.uniform(100, 200, w.T)], _clear_offsets(36, w.T))
    # both signs of A in every class: the sign alternates every five rows
    sign = np.where((np.arange(w.T) // 5) % 2 == 0, 1.0, -1.0)
    adv = sign * rng.uniform(0.2, 1.5, w.T)
    sup = lay.mask != 0
    clipped = sup & (cls != 4)
    for c in range(5):
        for sgn in (1.0, -1.0):
            assert (sup & (cls == c) & (sign == sgn)).any(), (c, sgn)
    weights = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask).astype(np.float32)
    for everything_clipped in (False, True):
        rr = np.where(cls == 4, 30.0 * sign, r) if everything_clipped else r
        logp_old = (lp_ref - rr).astype(np.float32)
        logp_teacher = (logp_old.astype(np.float64) + adv).astype(np.float32)
        r32 = lp_ref - logp_old.astype(np.float64)  # the log-ratio after the fp32 rounding of logp_old
        far = np.abs(np.abs(r32) - 20.0) >= 0.5
        assert far[sup].all()
        loss, lp, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, lay.mask, weights)
        ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                                   lay.mask, weights.astype(np.float64), w.tau)
        assert np.isfinite(loss).all() and np.isfinite(dH).all() and np.isfinite(dW).all()
        _close(lp[sup], ref.logp_s[sup], 1e-4, 1e-4, "logp")
        _close(loss, ref.loss, 1e-4, 2e-3, "loss")
        A = logp_teacher.astype(np.float64) - logp_old.astype(np.float64)
        hi, lo = sup & (r32 > 20), sup & (r32 < -20)
        _close(loss[hi & (A < 0)], -oracle_mod.KAPPA * A[hi & (A < 0)], 1e-4, 2e-3, "dual clip, r > 20")
        _close(loss[hi & (A > 0)], -(1 + oracle_mod.DELTA) * A[hi & (A > 0)], 1e-4, 2e-3, "ratio clip, r > 20")
        _close(loss[lo & (A < 0)], -(1 - oracle_mod.DELTA) * A[lo & (A < 0)], 1e-4, 2e-3, "ratio clip, r < -20")
        _close(loss[lo & (A > 0)], np.zeros(int((lo & (A > 0)).sum())), 1e-4, 0, "r < -20, A > 0")
        rows_clipped = sup & (np.abs(r32) > 20)
        assert (dH[rows_clipped] == 0).all() and (ref.dH_s[rows_clipped] == 0).all()
        assert (dH[~sup] == 0).all() and (loss[~sup] == 0).all()
        if everything_clipped:
            assert rows_clipped[sup].all()
            assert (dH == 0).all() and (dW == 0).all()
            assert (ref.dW_s == 0).all()
        else:
            assert clipped.sum() > 0 and (sup & ~clipped).sum() > 0
            assert _rel(dH, ref.dH_s) <= 1e-2, _rel(dH, ref.dH_s)
            assert _rel(dW, ref.dW_s) <= 1e-2, _rel(dW, ref.dW_s)


def _random_cases(n, seed=4049):
    rng = np.random.default_rng(seed)
    return [dict(T=int(rng.integers(1, 600)), d_s=8 * int(rng.integers(1, 41)), V=int(rng.integers(2, 5000)),
                 tau=float(rng.choice([0.4, 1.0, 1.7])), density=float(rng.uniform(0.1, 1.0)),
                 tiling=["bn256/cta1", "pair256/pair"][i % 2], seed=200 + i) for i in range(n)]


def _score_and_surrogate_check(lib, oracle_mod, w, mask, seed):
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    sup = mask != 0
    lse, lp = _score(lib, w, x["H_s"], x["W_s"], tokens, mask)
    ref_lse, ref_lp = oracle_mod.score(Hs, Ws, tokens, w.tau, rows=np.flatnonzero(sup))
    _close(lse[sup], ref_lse, 1e-4, 1e-4, "lse")
    _close(lp[sup], ref_lp, 1e-4, 1e-4, "logp")
    _, lp_full = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = (lp_full - _clear_offsets(seed, w.T)).astype(np.float32)
    adv = np.random.default_rng(seed + 1).choice([-1.0, 1.0], w.T) * \
        np.random.default_rng(seed + 2).uniform(0.2, 1.5, w.T)
    logp_teacher = (logp_old.astype(np.float64) + adv).astype(np.float32)
    weights = np.where(sup, 1.0 / int(sup.sum()), 0.0).astype(np.float32)
    loss, _, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, mask, weights)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               mask, weights.astype(np.float64), w.tau)
    _close(loss, ref.loss, 1e-4, 2e-3, "loss")
    assert _rel(dH, ref.dH_s) <= 1e-2, _rel(dH, ref.dH_s)
    assert _rel(dW, ref.dW_s) <= 1e-2, _rel(dW, ref.dW_s)


@pytest.mark.parametrize("case", _random_cases(8), ids=lambda c: f"T{c['T']}-d{c['d_s']}-V{c['V']}")
def test_surrogate_and_scoring_random_shapes(lib, oracle_mod, case, monkeypatch):
    fused, gemm = case["tiling"].split("/")
    monkeypatch.setenv("OPD_KL_FUSED", fused)
    monkeypatch.setenv("OPD_KL_GEMM", gemm)
    w = _case(T=case["T"], d_s=case["d_s"], V=case["V"], tau=case["tau"], n_traj=1, traj_len=case["T"],
              seed=case["seed"])
    mask = (np.random.default_rng(case["seed"]).random(w.T) < case["density"]).astype(np.uint8)
    mask[0] = 1
    _score_and_surrogate_check(lib, oracle_mod, w, mask, case["seed"])


@pytest.mark.parametrize("R", [1, 100, 128, 129, 300])
def test_surrogate_and_scoring_half_height_last_tile(lib, oracle_mod, monkeypatch, R):
    """The single-head kernels on CTA pairs with a last row tile of at most 128 supervised
    rows (R = 1, 100, 128, 300) run it as M = 128 MMAs; R = 129 does not. V = 2,100 leaves 52
    columns in the last vocabulary tile."""
    monkeypatch.setenv("OPD_KL_FUSED", "pair256")
    monkeypatch.setenv("OPD_KL_GEMM", "pair")
    w = _case(T=360, d_s=136, V=2100, tau=0.8, n_traj=1, traj_len=360, seed=41)
    mask = np.zeros(w.T, np.uint8)
    mask[np.random.default_rng(R).choice(w.T, R, replace=False)] = 1
    _score_and_surrogate_check(lib, oracle_mod, w, mask, 41 + R)


def test_surrogate_on_policy_and_accumulate(lib, oracle_mod):
    # rho = 1: the surrogate's gradient is the policy gradient -A (1[k = x] - p) / tau
    w = _case(T=300, d_s=128, V=2048, tau=1.0, n_traj=3, seed=33)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    _, lp_ref = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = lp_ref.astype(np.float32)
    logp_teacher = (lp_ref + 0.5).astype(np.float32)
    weights = np.ones(w.T, np.float32)
    init = torch.randn(w.V, w.d_s, device="cuda", generator=torch.Generator("cuda").manual_seed(1))
    loss, lp, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, lay.mask, weights, True, init)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               lay.mask, weights.astype(np.float64), w.tau)
    sup = lay.mask != 0
    _close(loss[sup], -0.5 * np.ones(sup.sum()), 1e-3, 0, "on-policy loss")
    assert _rel(dW - init.cpu().numpy(), ref.dW_s) <= 1e-2
    assert _rel(dH, ref.dH_s) <= 1e-2


def test_out_of_range_token_is_reported_not_read(lib):
    w = _case(T=256, d_s=64, V=500, n_traj=2, traj_len=128, seed=34)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    tokens[np.flatnonzero(lay.mask)[3]] = w.V + 7
    prob = lib.make_problem(w.T, w.d_s, w.d_s, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    lse = torch.empty(w.T, device="cuda")
    lp = torch.empty(w.T, device="cuda")
    lib.opd_score_tokens(prob, x["H_s"], x["W_s"], torch.from_numpy(tokens).cuda(),
                         torch.from_numpy(lay.mask).cuda(), lse, lp, ws)
    assert lib.opd_kl_get_status(ws) == lib.OPD_ERR_INVALID_ARG
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK


@pytest.mark.parametrize("name", ["qwen3_0p6b", "qwen3_1p7b", "qwen3_4b", "ragged_multiturn"])
def test_full_size_surrogate_and_scoring_sampled_rows(lib, oracle_mod, name):
    w = synth.WORKLOADS[name]
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    sup = np.flatnonzero(lay.mask)
    pick = np.unique(np.concatenate([sup[np.linspace(0, len(sup) - 1, 12).astype(int)], sup[:1], sup[-1:]]))
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    Ht, Wt = synth.host_values(x["H_t"]), synth.host_values(x["W_t"])
    # teacher scoring at full size
    lse_t, lp_t = _score(lib, w, x["H_t"], x["W_t"], tokens, lay.mask)
    ref_lse, ref_lp = oracle_mod.score(Ht, Wt, tokens, w.tau, rows=pick)
    _close(lse_t[pick], ref_lse, 1e-4, 1e-4, "teacher lse")
    _close(lp_t[pick], ref_lp, 1e-4, 1e-4, "teacher logp")
    # surrogate: synthetic teacher and behaviour log-probabilities, independent of the student
    # (wide ratio spread; a fp32 / fp64 branch flip needs a token within ~1e-5 of a kink)
    rng = np.random.default_rng(5)
    logp_teacher = rng.normal(-7.0, 1.0, w.T).astype(np.float32)
    logp_old = (logp_teacher.astype(np.float64) + rng.normal(0.0, 1.0, w.T)).astype(np.float32)
    weights = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask).astype(np.float32)
    loss, lp, dH, dW = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, lay.mask, weights)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                               lay.mask, weights.astype(np.float64), w.tau, rows=pick, want_dW=False)
    _close(lp[pick], ref.logp_s, 1e-4, 1e-4, "student logp")
    _close(loss[pick], ref.loss, 1e-4, 2e-3, "loss")
    assert _rel(dH[pick], ref.dH_s) <= 1e-2, _rel(dH[pick], ref.dH_s)
    # dW_s with only a few supervised rows at full shape
    mask2 = np.zeros_like(lay.mask)
    mask2[pick[::2]] = 1
    _, _, _, dW2 = _surrogate(lib, w, x, tokens, logp_old, logp_teacher, mask2, weights)
    ref2 = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), logp_teacher.astype(np.float64),
                                mask2, weights.astype(np.float64), w.tau, rows=pick[::2], want_dH=False)
    assert _rel(dW2, ref2.dW_s) <= 1e-2, _rel(dW2, ref2.dW_s)


def test_surrogate_loss_step_in_a_cuda_graph(lib):
    """The whole surrogate loss step (weights on the device, surrogate forward and backward,
    batch loss) makes no host synchronisation, so it captures into one CUDA graph; a replay
    reproduces the eager step."""
    w = _case(T=600, d_s=128, V=3000, tau=1.0, n_traj=6, traj_len=100, seed=43)
    lay = synth.layout(w)
    n_ids = int(lay.seg_id.max()) + 1
    x = synth.hidden_and_heads(w, "cuda")
    tokens = torch.from_numpy(synth.token_ids(w.seed, w.T, w.V)).cuda()
    rng = np.random.default_rng(43)
    logp_teacher = torch.from_numpy((rng.standard_normal(w.T) - 7.0).astype(np.float32)).cuda()
    logp_old = logp_teacher + torch.from_numpy((0.3 * rng.standard_normal(w.T)).astype(np.float32)).cuda()
    mask = torch.from_numpy(lay.mask).cuda()
    seg = torch.from_numpy(lay.seg_id).cuda()
    prob = lib.make_problem(w.T, w.d_s, w.d_s, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    seq_ws = torch.empty(lib.opd_seq_mean_token_mean_workspace_size(n_ids), dtype=torch.uint8, device="cuda")
    wts = torch.empty(w.T, device="cuda")
    loss = torch.empty(w.T, device="cuda")
    lp = torch.empty(w.T, device="cuda")
    dH = torch.empty(w.T, w.d_s, device="cuda")
    dW = torch.empty(w.V, w.d_s, device="cuda")
    total = torch.empty(1, device="cuda")

    def step():
        lib.opd_seq_mean_token_mean_device(seg, mask, n_ids, 1e-8, None, wts, None, seq_ws)
        lib.opd_surrogate_fwd_bwd(prob, x["H_s"], x["W_s"], tokens, logp_old, logp_teacher, mask, wts, loss, lp,
                                  dH, dW, False, ws)
        lib.opd_seq_mean_token_mean_device(seg, mask, n_ids, 1e-8, loss, None, total, seq_ws)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # eager step, outside the capture (kernel attributes are set here)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK and lib.opd_kl_get_status(seq_ws) == lib.OPD_OK
    eager = {k: v.clone() for k, v in dict(loss=loss, lp=lp, dH=dH, dW=dW, total=total).items()}
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for t in (loss, lp, dH, dW, total):
        t.fill_(float("nan"))
    graph.replay()
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK and lib.opd_kl_get_status(seq_ws) == lib.OPD_OK
    for k in ("loss", "lp", "dW"):
        np.testing.assert_array_equal(dict(loss=loss, lp=lp, dW=dW)[k].cpu().numpy(), eager[k].cpu().numpy())
    # dH_s: split-K partial sums in arrival order; L: a double sum over blocks in arrival order
    assert _rel(dH.cpu().numpy(), eager["dH"].cpu().numpy().astype(np.float64)) < 1e-5
    assert np.isfinite(total.item()) and abs(total.item() - eager["total"].item()) <= 1e-6 * abs(eager["total"].item())


def test_surrogate_and_scoring_with_every_row_masked(lib):
    """R = 0 with T > 0: zeros out, dW_s zeroed (or left as it was when accumulating), status OK."""
    w = _case(T=300, d_s=64, V=700, n_traj=3, traj_len=100, seed=44)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    mask = np.zeros(w.T, np.uint8)
    lse, lp = _score(lib, w, x["H_s"], x["W_s"], tokens, mask)
    assert (lse == 0).all() and (lp == 0).all()
    zeros = np.zeros(w.T, np.float32)
    loss, lp2, dH, dW = _surrogate(lib, w, x, tokens, zeros - 5.0, zeros - 4.0, mask, zeros + 1.0)
    assert (loss == 0).all() and (lp2 == 0).all() and (dH == 0).all() and (dW == 0).all()
    init = torch.full((w.V, w.d_s), 3.0, device="cuda")
    _, _, _, dW2 = _surrogate(lib, w, x, tokens, zeros - 5.0, zeros - 4.0, mask, zeros + 1.0, True, init)
    assert (dW2 == 3.0).all()
