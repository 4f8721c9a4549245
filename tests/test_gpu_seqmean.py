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
