"""The torch.autograd entry points: gradients through .backward() equal the C ABI's results
(and, through them, the oracle's, which the other parity tests establish)."""

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def mods():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import autograd, opd_kl
    return autograd, opd_kl


def _rel(a, b):
    a, b = np.asarray(a, np.float64), np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_reverse_kl_autograd_matches_abi_and_oracle(mods, oracle_mod, name):
    ag, lib = mods
    if name == "tiny_fp32":
        w = synth.WORKLOADS["tiny_fp32"]
    else:
        w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="small", T=400, d_s=128, d_t=192, V=900, tau=0.9,
                         n_traj=4, traj_len=100, seed=51)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    H_s = x["H_s"].clone().requires_grad_(True)
    W_s = x["W_s"].clone().requires_grad_(True)
    mask = torch.from_numpy(lay.mask).cuda()
    g = torch.from_numpy(synth.uniform_weights(w.seed, w.T).astype(np.float32)).cuda()
    kl = ag.OPDReverseKL.apply(H_s, x["H_t"], W_s, x["W_t"], mask, w.tau)
    (kl * g).sum().backward()
    gg = np.where(lay.mask != 0, g.cpu().numpy().astype(np.float64), 0.0)
    ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), lay.mask, gg, w.tau)
    tol = 1e-4 if w.dtype == "f32" else 1e-2
    assert np.abs(kl.detach().cpu().numpy() - ref.kl).max() <= 1e-4 + 2e-3 * np.abs(ref.kl).max()
    # bf16 inputs get bf16 gradients (autograd's dtype rule): one more rounding, still inside 1e-2
    assert _rel(H_s.grad.float().cpu().numpy(), ref.dH_s) <= tol
    assert _rel(W_s.grad.float().cpu().numpy(), ref.dW_s) <= tol


def test_seq_mean_loss_autograd(mods, oracle_mod):
    ag, lib = mods
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="small", T=500, d_s=128, d_t=128, V=700, tau=1.0,
                     n_traj=5, traj_len=100, seed=52)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    H_s = x["H_s"].clone().requires_grad_(True)
    W_s = x["W_s"].clone().requires_grad_(True)
    n_ids = int(lay.seg_id.max()) + 1
    loss = ag.OPDSeqMeanKLLoss.apply(H_s, x["H_t"], W_s, x["W_t"], torch.from_numpy(lay.mask).cuda(),
                                     torch.from_numpy(lay.seg_id).cuda(), n_ids, w.tau)
    (2.0 * loss).backward()
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
    ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), lay.mask, 2.0 * g,
                            w.tau)
    want = float(np.dot(g, ref.kl))
    assert abs(float(loss.detach()) - want) <= 1e-4 + 2e-3 * abs(want)
    assert _rel(H_s.grad.float().cpu().numpy(), ref.dH_s) <= 1e-2
    assert _rel(W_s.grad.float().cpu().numpy(), ref.dW_s) <= 1e-2


def test_surrogate_loss_autograd_and_scoring(mods, oracle_mod):
    """OPDSurrogateLoss (device seq-mean-token-mean weights, one surrogate call) and score_tokens
    against the oracle: the loss, the teacher's scores, and the gradients through .backward()."""
    ag, lib = mods
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="small", T=500, d_s=128, d_t=192, V=900, tau=1.0,
                     n_traj=5, traj_len=100, seed=53)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    tokens = synth.token_ids(w.seed, w.T, w.V)
    tok = torch.from_numpy(tokens).cuda()
    mask = torch.from_numpy(lay.mask).cuda()
    # the teacher's scores of the sampled tokens, then a behaviour policy near the student
    lse_t, lp_t = ag.score_tokens(x["H_t"], x["W_t"], tok, mask, w.tau)
    Ht, Wt = synth.host_values(x["H_t"]), synth.host_values(x["W_t"])
    sup = lay.mask != 0
    ref_lse, ref_lp = oracle_mod.score(Ht, Wt, tokens, w.tau, rows=np.flatnonzero(sup))
    assert np.abs(lse_t.cpu().numpy()[sup] - ref_lse).max() <= 1e-4 + 1e-4 * np.abs(ref_lse).max()
    assert np.abs(lp_t.cpu().numpy()[sup] - ref_lp).max() <= 1e-4 + 1e-4 * np.abs(ref_lp).max()
    # both sides get the same inputs, none of them from the GPU: the teacher's log-probabilities
    # from the oracle, a behaviour policy within 5% of the student (no ratio clip is active)
    _, lp_teacher = oracle_mod.score(Ht, Wt, tokens, w.tau)
    lp_teacher = lp_teacher.astype(np.float32)
    Hs, Ws = synth.host_values(x["H_s"]), synth.host_values(x["W_s"])
    _, lp_s = oracle_mod.score(Hs, Ws, tokens, w.tau)
    logp_old = (lp_s + np.random.default_rng(53).uniform(-0.05, 0.05, w.T)).astype(np.float32)
    H_s = x["H_s"].clone().requires_grad_(True)
    W_s = x["W_s"].clone().requires_grad_(True)
    n_ids = int(lay.seg_id.max()) + 1
    loss = ag.OPDSurrogateLoss.apply(H_s, W_s, tok, torch.from_numpy(logp_old).cuda(),
                                     torch.from_numpy(lp_teacher).cuda(), mask, torch.from_numpy(lay.seg_id).cuda(),
                                     n_ids, w.tau)
    (3.0 * loss).backward()
    wts = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
    ref = oracle_mod.surrogate(Hs, Ws, tokens, logp_old.astype(np.float64), lp_teacher.astype(np.float64),
                               lay.mask, 3.0 * wts, w.tau)
    want = float(np.dot(wts, ref.loss))
    assert abs(float(loss.detach()) - want) <= 1e-4 + 2e-3 * abs(want)
    assert _rel(H_s.grad.float().cpu().numpy(), ref.dH_s) <= 1e-2
    assert _rel(W_s.grad.float().cpu().numpy(), ref.dW_s) <= 1e-2


def test_debug_mode_raises_on_bad_ids_through_autograd(mods, monkeypatch):
    """The autograd functions do not read the device status word; with OPD_KL_SYNC_CHECK=1 the
    library itself synchronises after each call and the binding raises OpdError. A token id past
    the vocabulary (scoring) and a response id past n_ids (the surrogate's weights) are reported
    that way; without debug mode the same calls return."""
    ag, lib = mods
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="dbg", T=256, d_s=64, d_t=64, V=500, tau=1.0,
                     n_traj=2, traj_len=128, seed=53)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    mask = torch.from_numpy(lay.mask).cuda()
    tokens = torch.from_numpy(synth.token_ids(w.seed, w.T, w.V)).cuda()
    bad_tokens = tokens.clone()
    bad_tokens[int(np.flatnonzero(lay.mask)[0])] = w.V + 3
    seg = torch.from_numpy(lay.seg_id).cuda()
    n_ids = int(lay.seg_id.max()) + 1
    bad_seg = seg.clone()
    bad_seg[int(np.flatnonzero(lay.seg_id >= 0)[0])] = n_ids + 5
    lp = torch.full((w.T,), -6.0, device="cuda")
    ag.score_tokens(x["H_s"], x["W_s"], bad_tokens, mask)  # outside debug mode: returns
    ag.OPDSurrogateLoss.apply(x["H_s"], x["W_s"], tokens, lp, lp + 0.5, mask, bad_seg, n_ids, 1.0, 1e-8)
    torch.cuda.synchronize()
    monkeypatch.setenv("OPD_KL_SYNC_CHECK", "1")
    with pytest.raises(lib.OpdError) as e1:
        ag.score_tokens(x["H_s"], x["W_s"], bad_tokens, mask)
    assert e1.value.status == lib.OPD_ERR_INVALID_ARG
    with pytest.raises(lib.OpdError) as e2:
        ag.OPDSurrogateLoss.apply(x["H_s"], x["W_s"], tokens, lp, lp + 0.5, mask, bad_seg, n_ids, 1.0, 1e-8)
    assert e2.value.status == lib.OPD_ERR_INVALID_ARG
    # good ids in debug mode: no error
    ag.score_tokens(x["H_s"], x["W_s"], tokens, mask)
