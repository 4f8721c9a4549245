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
