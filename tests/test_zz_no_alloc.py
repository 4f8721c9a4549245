"""The workspace-free forward entry point against the oracle and the regular forward.

opd_kl_forward_noalloc serves callers that may not allocate device memory at
all, such as a host process that owns the whole GPU through its own fixed pool
and forbids libraries from calling cudaMalloc. It keeps its scratch in a fixed
array inside the library instead of a caller-provided workspace. This file
checks it through the C ABI against the float64 oracle and against
opd_kl_forward, with the same tolerance as the parity tests, on three calls in a
row with different problems (each call reuses the array the previous one left
behind). It runs last so that a failure here leaves every other test already run.
"""

import numpy as np
import pytest
import torch

from paper_2609_36608_gb300 import synth

pytestmark = pytest.mark.gpu

KL_ABS, KL_REL = 1e-4, 2e-3


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl
    return opd_kl


def _case(name, **kw):
    base = dict(name=name, d_s=256, d_t=384, V=1000, tau=0.7, traj_len=100, n_traj=1)
    base.update(kw)
    return synth.scaled(synth.WORKLOADS["qwen3_1p7b"], **base)


def _both(lib, w):
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    mask = torch.from_numpy(lay.mask).cuda()
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    kl_ref = torch.full((w.T,), float("nan"), device="cuda")
    st_ref = torch.full((w.T, 3), float("nan"), device="cuda")
    lib.opd_kl_forward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, kl_ref, st_ref, ws)
    kl = torch.full((w.T,), float("nan"), device="cuda")
    st = torch.full((w.T, 3), float("nan"), device="cuda")
    lib.opd_kl_forward_noalloc(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, kl, st)
    torch.cuda.synchronize()
    return lay.mask != 0, kl.cpu().numpy(), st.cpu().numpy(), kl_ref.cpu().numpy(), st_ref.cpu().numpy()


def test_noalloc_forward_matches_oracle_and_workspace_forward_on_three_calls(lib, oracle_mod):
    # every row is scheduled here (no compaction): T = 300 leaves a last row tile of 44 rows,
    # which runs at half height on a CTA pair
    cases = [_case("noalloc_a", T=700, seed=21),
             _case("noalloc_b", T=lib.OPD_KL_NOALLOC_MAX_ROWS, d_s=128, d_t=192, V=1237, tau=1.0, seed=22,
                   traj_len=512),
             _case("noalloc_c", T=300, d_s=192, d_t=256, V=3000, tau=1.3, seed=23, traj_len=300)]
    for w in cases:
        sup, kl, st, kl_ref, st_ref = _both(lib, w)
        # against the float64 oracle, on every supervised row
        x = synth.hidden_and_heads(w, "cuda")
        rows = np.flatnonzero(sup)
        ref = oracle_mod.opd_kl(*(synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")), sup,
                                np.zeros(w.T), w.tau, rows=rows, want_dH=False, want_dW=False)
        excess = np.abs(kl[rows] - ref.kl) - (KL_ABS + KL_REL * np.abs(ref.kl))
        assert excess.max() <= 0, (w.name, "oracle", float(excess.max()))
        for col, want in ((0, ref.lse_s), (1, ref.lse_t), (2, ref.kl)):
            tol = 1e-4 + (KL_REL if col == 2 else 1e-5) * np.abs(want)
            assert (np.abs(st[rows, col] - want) <= tol).all(), (w.name, "stats column", col)
        # against the workspace forward
        excess = np.abs(kl - kl_ref) - (KL_ABS + KL_REL * np.abs(kl_ref))
        assert excess.max() <= 0, (w.name, float(excess.max()))
        assert (kl[~sup] == 0).all() and (st[~sup] == 0).all()
        np.testing.assert_allclose(st[sup], st_ref[sup], rtol=1e-5, atol=1e-4)


def test_noalloc_rejects_rows_beyond_its_fixed_scratch(lib):
    T = lib.OPD_KL_NOALLOC_MAX_ROWS + 1
    prob = lib.make_problem(T, 64, 64, 128, lib.OPD_DTYPE_BF16, 1.0)
    H = torch.zeros(T, 64, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    mask = torch.ones(T, dtype=torch.uint8, device="cuda")
    out = torch.empty(T, device="cuda")
    stats = torch.empty(T, 3, device="cuda")
    with pytest.raises(lib.OpdError) as e:
        lib.opd_kl_forward_noalloc(prob, H, H, W, W, mask, out, stats)
    assert e.value.status == lib.OPD_ERR_UNSUPPORTED
