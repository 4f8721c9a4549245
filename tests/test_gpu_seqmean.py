"""GPU parity of the on-device seq-mean-token-mean (Appendix B.4, Eq. opd-surrogate)
against the oracle's helper: per-token weights, and the weighted loss sum_i w_i l_i."""

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl
    return opd_kl


@pytest.mark.parametrize("name", ["tiny_fp32", "qwen3_1p7b", "ragged_multiturn"])
def test_weights_and_loss_match_oracle(lib, oracle_mod, name):
    lay = synth.layout(synth.WORKLOADS[name])
    T = len(lay.mask)
    n_ids = int(lay.seg_id.max()) + 1
    seg = torch.from_numpy(lay.seg_id).cuda()
    mask = torch.from_numpy(lay.mask).cuda()
    loss = np.random.default_rng(0).standard_normal(T).astype(np.float32)
    w_out = torch.full((T,), float("nan"), device="cuda")
    l_out = torch.full((1,), float("nan"), device="cuda")
    ws = lib.opd_seq_mean_token_mean_device(seg, mask, n_ids, 1e-8, torch.from_numpy(loss).cuda(), w_out, l_out)
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    ref = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
    np.testing.assert_allclose(w_out.cpu().numpy(), ref, rtol=1e-6, atol=0)
    want = float(np.dot(ref, loss.astype(np.float64)))
    assert abs(float(l_out.item()) - want) <= 1e-6 * max(1.0, abs(want))


def test_response_id_out_of_range_is_reported(lib):
    seg = torch.tensor([0, 0, 1, 5, -1], dtype=torch.int32, device="cuda")
    mask = torch.ones(5, dtype=torch.uint8, device="cuda")
    w_out = torch.empty(5, device="cuda")
    ws = lib.opd_seq_mean_token_mean_device(seg, mask, 2, 1e-8, None, w_out, None)
    assert lib.opd_kl_get_status(ws) == lib.OPD_ERR_INVALID_ARG


def _seq_mean_step(lib, w, x, lay, n_ids=None, accumulate=False, dW_init=None):
    dtype = lib.OPD_DTYPE_F32 if w.dtype == "f32" else lib.OPD_DTYPE_BF16
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, dtype, w.tau)
    n_ids = int(lay.seg_id.max()) + 1 if n_ids is None else n_ids
    ws = lib.allocate_seq_mean_workspace(prob, n_ids, "cuda")
    loss = torch.full((1,), float("nan"), device="cuda")
    kl = torch.full((w.T,), float("nan"), device="cuda")
    stats = torch.full((w.T, 3), float("nan"), device="cuda")
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    dW = torch.full((w.V, w.d_s), float("nan"), device="cuda") if dW_init is None else dW_init.clone()
    lib.opd_kl_seq_mean_fwd_bwd(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], torch.from_numpy(lay.mask).cuda(),
                                torch.from_numpy(lay.seg_id).cuda(), n_ids, 1e-8, loss, kl, stats, dH, dW,
                                accumulate, ws)
    torch.cuda.synchronize()
    return ws, float(loss.item()), kl.cpu().numpy(), dH.cpu().numpy(), dW.cpu().numpy()


def _rel(a, b):
    return float(np.linalg.norm(np.asarray(a, np.float64) - b) / max(np.linalg.norm(b), 1e-300))


@pytest.mark.parametrize("case", ["tiny_fp32", "small_bf16"])
def test_kl_seq_mean_step_matches_oracle(lib, oracle_mod, case):
    """One call: device weights, forward with L summed in the combine pass, backward with g = w."""
    if case == "tiny_fp32":
        w = synth.WORKLOADS["tiny_fp32"]
        kl_tol, grad_tol = (1e-5, 1e-5), 1e-4
    else:
        w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="small", T=700, d_s=256, d_t=384, V=1237, tau=0.8,
                         n_traj=7, traj_len=100, seed=41)
        kl_tol, grad_tol = (1e-4, 2e-3), 1e-2
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    ws, L, kl, dH, dW = _seq_mean_step(lib, w, x, lay)
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    g = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
    ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), lay.mask, g, w.tau)
    excess = np.abs(kl - ref.kl) - (kl_tol[0] + kl_tol[1] * np.abs(ref.kl))
    assert excess.max() <= 0
    want = float(np.dot(g, ref.kl))  # sum_i w_i KL_i, with sum_i w_i = 1
    assert abs(L - want) <= kl_tol[0] + kl_tol[1] * abs(want), (L, want)
    assert _rel(dH, ref.dH_s) <= grad_tol and _rel(dW, ref.dW_s) <= grad_tol


def test_kl_seq_mean_step_full_size_agrees_with_two_calls(lib):
    """At the Qwen3-1.7B-shaped size: the one-call loss step gives the same KL and gradients as
    opd_kl_fwd_bwd with the host helper's weights, and L is the weighted sum of its own KL."""
    w = synth.WORKLOADS["qwen3_1p7b"]
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    ws, L, kl, dH, dW = _seq_mean_step(lib, w, x, lay)
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    g = lib.opd_seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws2 = lib.allocate_workspace(prob, "cuda")
    kl2, st2 = torch.empty(w.T, device="cuda"), torch.empty(w.T, 3, device="cuda")
    dH2, dW2 = torch.empty(w.T, w.d_s, device="cuda"), torch.empty(w.V, w.d_s, device="cuda")
    lib.opd_kl_fwd_bwd(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], torch.from_numpy(lay.mask).cuda(),
                       torch.from_numpy(g).cuda(), kl2, st2, dH2, dW2, False, ws2)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(kl, kl2.cpu().numpy())
    assert _rel(dH, dH2.cpu().numpy().astype(np.float64)) < 1e-5
    assert _rel(dW, dW2.cpu().numpy().astype(np.float64)) < 1e-5
    want = float(np.dot(g.astype(np.float64), kl.astype(np.float64)))
    assert abs(L - want) <= 1e-6 * max(1.0, abs(want))


def test_kl_seq_mean_step_bad_response_id(lib):
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="small", T=300, d_s=64, d_t=64, V=500, n_traj=3,
                     traj_len=100, seed=42)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    ws, *_ = _seq_mean_step(lib, w, x, lay, n_ids=1)  # ids 1, 2, ... are out of range
    assert lib.opd_kl_get_status(ws) == lib.OPD_ERR_INVALID_ARG
