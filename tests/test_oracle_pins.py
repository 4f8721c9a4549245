"""Pins for the float64 CPU oracle, checked against what the definition fixes.

The paper prints no numeric example for the per-token reverse KL, so the oracle
is pinned by facts that do not depend on its own code: closed forms (uniform
teacher, two-token vocabulary, a hand-derived three-token example), invariants
(identical policies, non-negativity, zero-sum gradient rows, masking, logit
shifts, logit scaling, row permutation, linearity in the upstream weights),
central finite differences, and a float64 PyTorch autograd evaluation of the
same loss. Each plausible slip (forward instead of reverse KL, a missing 1/tau,
a dropped -KL term, a sign or transposition error, masked rows leaking into
dW_s) fails at least one test here.

Definitions: ActFirst-OPD Section 3, Eq. opd-objective and Eq. reverse-kl;
Appendix B.4 (mask, frozen teacher, seq-mean-token-mean).
"""

import math
import os

import numpy as np
import pytest
import scipy.special as sp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _problem(seed, T=7, d_s=5, d_t=6, V=13, std=2.0, mask=None):
    rng = np.random.default_rng(seed)
    H_s = rng.standard_normal((T, d_s)).astype(np.float32)
    H_t = rng.standard_normal((T, d_t)).astype(np.float32)
    W_s = (rng.standard_normal((V, d_s)) * std / math.sqrt(d_s)).astype(np.float32)
    W_t = (rng.standard_normal((V, d_t)) * std / math.sqrt(d_t)).astype(np.float32)
    if mask is None:
        mask = (rng.random(T) < 0.7).astype(np.uint8)
        mask[0] = 1
    g = rng.uniform(0.5, 1.5, T)
    return H_s, H_t, W_s, W_t, np.asarray(mask, np.uint8), g


def _loss(o, H_s, H_t, W_s, W_t, mask, g, tau):
    r = o.opd_kl(H_s, H_t, W_s, W_t, mask, g, tau, want_dH=False, want_dW=False)
    return float(np.dot(g, r.kl))


def _read_golden(name):
    vals = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *rest = line.split()
            vals[key] = [float(x) for x in rest]
    return vals


def test_student_equals_teacher_gives_zero(oracle_mod):
    H_s, _, W_s, _, mask, g = _problem(1, d_s=6, d_t=6)
    r = oracle_mod.opd_kl(H_s, H_s, W_s, W_s, mask, g, 1.3, want_dZ=True)
    assert np.abs(r.kl).max() < 1e-14
    assert np.abs(r.dZ).max() < 1e-14
    assert np.abs(r.dH_s).max() < 1e-13
    assert np.abs(r.dW_s).max() < 1e-13


def test_kl_nonnegative_and_positive_when_policies_differ(oracle_mod):
    for seed in range(5):
        H_s, H_t, W_s, W_t, mask, g = _problem(10 + seed)
        r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0)
        assert (r.kl >= 0).all()
        assert (r.kl[mask == 1] > 1e-6).all()


def test_gradient_rows_sum_to_zero(oracle_mod):
    # sum_k p_s[k](lp_s - lp_t - KL) = KL - KL = 0
    H_s, H_t, W_s, W_t, mask, g = _problem(2, V=50)
    r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 0.8, want_dZ=True)
    row_sum = r.dZ.sum(axis=1)
    scale = np.abs(r.dZ).sum(axis=1) + 1e-300
    assert (np.abs(row_sum) <= 1e-14 * np.maximum(scale, 1.0)).all()
    assert (np.abs(r.dZ[mask == 1]).sum(axis=1) > 1e-4).all()


def test_masked_rows_contribute_nothing(oracle_mod):
    mask = np.array([1, 0, 1, 0, 0, 1, 1], np.uint8)
    H_s, H_t, W_s, W_t, _, g = _problem(3, mask=mask)
    a = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0, want_dZ=True)
    H_s2, H_t2 = H_s.copy(), H_t.copy()
    H_s2[mask == 0] = 7.0 * np.random.default_rng(9).standard_normal(H_s2[mask == 0].shape)
    H_t2[mask == 0] = -3.0
    g2 = g.copy()
    g2[mask == 0] = 123.0
    b = oracle_mod.opd_kl(H_s2, H_t2, W_s, W_t, mask, g2, 1.0, want_dZ=True)
    assert np.array_equal(a.kl, b.kl)
    assert np.array_equal(a.dW_s, b.dW_s)
    assert np.array_equal(a.dH_s[mask == 1], b.dH_s[mask == 1])
    assert (a.kl[mask == 0] == 0).all() and (a.dH_s[mask == 0] == 0).all()
    assert (a.dZ[mask == 0] == 0).all()


def test_uniform_teacher_closed_form(oracle_mod):
    # W_t = 0 makes the teacher uniform: KL(p || U) = log V - H(p),
    # dz = (g/tau) p (log p + H(p)).
    tau = 0.7
    H_s, H_t, W_s, W_t, mask, g = _problem(4, V=40)
    W_t = np.zeros_like(W_t)
    r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, tau, want_dZ=True)
    u = (H_s.astype(np.float64) @ W_s.astype(np.float64).T) / tau
    p = sp.softmax(u, axis=1)
    ent = sp.entr(p).sum(axis=1)
    V = W_s.shape[0]
    kl_ref = np.where(mask == 1, math.log(V) - ent, 0.0)
    np.testing.assert_allclose(r.kl, kl_ref, rtol=1e-12, atol=1e-14)
    dz_ref = (g / tau)[:, None] * p * (np.log(p) + ent[:, None]) * mask[:, None]
    np.testing.assert_allclose(r.dZ, dz_ref, rtol=1e-10, atol=1e-15)
    np.testing.assert_allclose(r.lse_t, math.log(V), rtol=0, atol=1e-14)


def test_two_token_vocabulary_bernoulli(oracle_mod):
    tau = 1.7
    H_s, H_t, W_s, W_t, mask, g = _problem(5, V=2, mask=np.ones(7, np.uint8))
    r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, tau, want_dZ=True)
    us = (H_s.astype(np.float64) @ W_s.astype(np.float64).T) / tau
    ut = (H_t.astype(np.float64) @ W_t.astype(np.float64).T) / tau
    p = sp.expit(us[:, 1] - us[:, 0])
    q = sp.expit(ut[:, 1] - ut[:, 0])
    kl = p * np.log(p / q) + (1 - p) * np.log((1 - p) / (1 - q))
    np.testing.assert_allclose(r.kl, kl, rtol=1e-11, atol=1e-15)
    # d KL / d (u1 - u0) = p (1-p) [log(p/q) - log((1-p)/(1-q))]; dz = g/tau times that
    dkl = p * (1 - p) * (np.log(p / q) - np.log((1 - p) / (1 - q)))
    np.testing.assert_allclose(r.dZ[:, 1], g / tau * dkl, rtol=1e-9, atol=1e-15)
    np.testing.assert_allclose(r.dZ[:, 0], -g / tau * dkl, rtol=1e-9, atol=1e-15)


def test_hand_worked_three_token_example(oracle_mod):
    gold = _read_golden("hand_v3.txt")
    ln2 = np.float32(math.log(2.0))
    H = np.ones((1, 1), np.float32)
    W_s = np.array([[0.0], [ln2], [0.0]], np.float32)
    W_t = np.array([[0.0], [0.0], [ln2]], np.float32)
    r = oracle_mod.opd_kl(H, H, W_s, W_t, np.ones(1, np.uint8), np.ones(1), 1.0, want_dZ=True)
    assert abs(r.kl[0] - gold["kl"][0]) < 1e-7
    assert abs(r.lse_s[0] - gold["lse_s"][0]) < 1e-7
    assert abs(r.lse_t[0] - gold["lse_t"][0]) < 1e-7
    for k in range(3):
        assert abs(r.dZ[0, k] - gold[f"dz{k}"][0]) < 1e-7
        assert abs(r.dW_s[k, 0] - gold[f"dz{k}"][0]) < 1e-7
    assert abs(r.dH_s[0, 0] - gold["dH"][0]) < 1e-7


def test_logit_shift_invariance(oracle_mod):
    # Appending a column with H[i, d] = a_i and W[k, d] = 1 adds a_i to every logit
    # of row i; softmax, KL and dz are unchanged.
    H_s, H_t, W_s, W_t, mask, g = _problem(6)
    a = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0, want_dZ=True)
    shift_s = np.arange(7, dtype=np.float32)[:, None] * 0.75 - 2.0
    shift_t = -np.arange(7, dtype=np.float32)[:, None] * 0.5 + 1.0
    H_s2 = np.concatenate([H_s, shift_s], axis=1)
    H_t2 = np.concatenate([H_t, shift_t], axis=1)
    W_s2 = np.concatenate([W_s, np.ones((W_s.shape[0], 1), np.float32)], axis=1)
    W_t2 = np.concatenate([W_t, np.ones((W_t.shape[0], 1), np.float32)], axis=1)
    b = oracle_mod.opd_kl(H_s2, H_t2, W_s2, W_t2, mask, g, 1.0, want_dZ=True)
    np.testing.assert_allclose(b.kl, a.kl, rtol=1e-11, atol=1e-14)
    np.testing.assert_allclose(b.dZ, a.dZ, rtol=1e-9, atol=1e-14)
    np.testing.assert_allclose(b.dW_s[:, :-1], a.dW_s, rtol=1e-9, atol=1e-13)


def test_temperature_scale_invariance(oracle_mod):
    # (W_s, W_t, tau) -> (c W_s, c W_t, c tau) keeps u = z / tau, so KL is unchanged;
    # dz (w.r.t. the raw logits) scales by 1/c, dH_s = dz W_s is unchanged, dW_s scales by 1/c.
    H_s, H_t, W_s, W_t, mask, g = _problem(7)
    c = 2.0
    a = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 0.9)
    b = oracle_mod.opd_kl(H_s, H_t, W_s * c, W_t * c, mask, g, 0.9 * c)
    np.testing.assert_allclose(b.kl, a.kl, rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(b.dH_s, a.dH_s, rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(b.dW_s * c, a.dW_s, rtol=1e-10, atol=1e-14)


def test_row_permutation(oracle_mod):
    H_s, H_t, W_s, W_t, mask, g = _problem(8, T=9)
    perm = np.random.default_rng(0).permutation(9)
    a = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0)
    b = oracle_mod.opd_kl(H_s[perm], H_t[perm], W_s, W_t, mask[perm], g[perm], 1.0)
    np.testing.assert_array_equal(b.kl, a.kl[perm])
    np.testing.assert_array_equal(b.dH_s, a.dH_s[perm])
    np.testing.assert_allclose(b.dW_s, a.dW_s, rtol=1e-12, atol=1e-15)


def test_backward_linear_in_upstream_weights(oracle_mod):
    H_s, H_t, W_s, W_t, mask, g1 = _problem(9)
    g2 = np.random.default_rng(1).uniform(-1, 1, g1.shape)
    r1 = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g1, 1.0)
    r2 = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g2, 1.0)
    r3 = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, 2.0 * g1 - 3.0 * g2, 1.0)
    np.testing.assert_array_equal(r3.kl, r1.kl)
    np.testing.assert_allclose(r3.dH_s, 2 * r1.dH_s - 3 * r2.dH_s, rtol=1e-10, atol=1e-14)
    np.testing.assert_allclose(r3.dW_s, 2 * r1.dW_s - 3 * r2.dW_s, rtol=1e-10, atol=1e-14)


@pytest.mark.parametrize("tau", [1.0, 0.7])
def test_finite_differences(oracle_mod, tau):
    # L = sum_i g_i KL_i; central differences in float64 on float64-exact inputs.
    # Perturbations are applied to float64 copies, so inputs are passed as float64
    # through a float32 round trip only where exact: use a wrapper that feeds the
    # oracle float32 arrays holding exactly representable perturbed values.
    H_s, H_t, W_s, W_t, mask, g = _problem(11, T=5, d_s=4, d_t=3, V=9)
    r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, tau)
    h = 2.0 ** -10  # exact in float32 when added to values of magnitude < 2^13 with enough bits
    rng = np.random.default_rng(3)
    for _ in range(12):
        i, j = rng.integers(0, 5), rng.integers(0, 4)
        Hp, Hm = H_s.copy(), H_s.copy()
        Hp[i, j] += np.float32(h)
        Hm[i, j] -= np.float32(h)
        step = float(Hp[i, j]) - float(Hm[i, j])
        fd = (_loss(oracle_mod, Hp, H_t, W_s, W_t, mask, g, tau)
              - _loss(oracle_mod, Hm, H_t, W_s, W_t, mask, g, tau)) / step
        assert abs(fd - r.dH_s[i, j]) <= 2e-5 * max(1.0, abs(fd)), (i, j, fd, r.dH_s[i, j])
        k, j = rng.integers(0, 9), rng.integers(0, 4)
        Wp, Wm = W_s.copy(), W_s.copy()
        Wp[k, j] += np.float32(h)
        Wm[k, j] -= np.float32(h)
        step = float(Wp[k, j]) - float(Wm[k, j])
        fd = (_loss(oracle_mod, H_s, H_t, Wp, W_t, mask, g, tau)
              - _loss(oracle_mod, H_s, H_t, Wm, W_t, mask, g, tau)) / step
        assert abs(fd - r.dW_s[k, j]) <= 2e-5 * max(1.0, abs(fd)), (k, j, fd, r.dW_s[k, j])


def test_torch_float64_autograd_cross_check(oracle_mod):
    torch = pytest.importorskip("torch")
    tau = 0.8
    H_s, H_t, W_s, W_t, mask, g = _problem(12, T=11, d_s=8, d_t=12, V=57)
    r = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, tau)
    hs = torch.tensor(H_s, dtype=torch.float64, requires_grad=True)
    ws = torch.tensor(W_s, dtype=torch.float64, requires_grad=True)
    ht = torch.tensor(H_t, dtype=torch.float64)
    wt = torch.tensor(W_t, dtype=torch.float64)
    lps = torch.log_softmax(hs @ ws.T / tau, dim=-1)
    lpt = torch.log_softmax(ht @ wt.T / tau, dim=-1)
    kl = torch.nn.functional.kl_div(lpt, lps, log_target=True, reduction="none").sum(-1)
    kl = kl * torch.tensor(mask, dtype=torch.float64)
    (kl * torch.tensor(g)).sum().backward()
    np.testing.assert_allclose(r.kl, kl.detach().numpy(), rtol=1e-11, atol=1e-14)
    np.testing.assert_allclose(r.dH_s, hs.grad.numpy(), rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(r.dW_s, ws.grad.numpy(), rtol=1e-9, atol=1e-13)


def test_bf16_bit_inputs_read_exactly(oracle_mod):
    H_s, H_t, W_s, W_t, mask, g = _problem(13)

    def to_bf16_bits(a):
        u = a.astype(np.float32).view(np.uint32)
        return (u >> 16).astype(np.uint16)  # truncation: the value is exactly a bf16 number

    bits = [to_bf16_bits(x) for x in (H_s, H_t, W_s, W_t)]
    vals = [(b.astype(np.uint32) << 16).view(np.float32) for b in bits]
    a = oracle_mod.opd_kl(*bits, mask, g, 1.0)
    b = oracle_mod.opd_kl(*vals, mask, g, 1.0)
    np.testing.assert_array_equal(a.kl, b.kl)
    np.testing.assert_array_equal(a.dH_s, b.dH_s)
    np.testing.assert_array_equal(a.dW_s, b.dW_s)


def test_row_subset_and_mask_subset_agree_with_full_run(oracle_mod):
    H_s, H_t, W_s, W_t, mask, g = _problem(14, T=10)
    full = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0)
    rows = np.flatnonzero(mask)[::2]
    sub = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0, rows=rows)
    np.testing.assert_array_equal(sub.kl, full.kl[rows])
    np.testing.assert_array_equal(sub.dH_s, full.dH_s[rows])
    m2 = np.zeros_like(mask)
    m2[rows] = 1
    only = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, m2, g, 1.0)
    np.testing.assert_allclose(sub.dW_s, only.dW_s, rtol=1e-13, atol=1e-16)


def test_seq_mean_token_mean_weights_golden(oracle_mod):
    gold = _read_golden("seq_mean_token_mean.txt")
    seg = np.array(gold["seg_id"], np.int32)
    mask = np.array(gold["mask"], np.uint8)
    w = oracle_mod.seq_mean_token_mean_weights(seg, mask, 1e-8)
    np.testing.assert_allclose(w, gold["w"], rtol=1e-15, atol=0)


def test_seq_mean_token_mean_matches_group_means(oracle_mod):
    # sum_i w_i l_i equals the mean over responses of each response's masked token mean.
    rng = np.random.default_rng(15)
    seg = np.repeat(np.arange(-1, 6), rng.integers(1, 9, 7)).astype(np.int32)
    mask = (rng.random(seg.shape[0]) < 0.6).astype(np.uint8)
    mask[seg < 0] = 0
    loss = rng.standard_normal(seg.shape[0])
    w = oracle_mod.seq_mean_token_mean_weights(seg, mask, 1e-8)
    ids = sorted(set(seg[seg >= 0].tolist()))
    per_resp = [(loss[(seg == b) & (mask == 1)].sum()) / ((mask[seg == b]).sum() + 1e-8) for b in ids]
    assert abs(np.dot(w, loss) - np.mean(per_resp)) < 1e-13


def test_invalid_arguments_are_rejected(oracle_mod):
    H_s, H_t, W_s, W_t, mask, g = _problem(16)
    with pytest.raises(ValueError):
        oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 0.0)
    with pytest.raises(ValueError):
        oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask, g, 1.0, rows=[0, 99])
    with pytest.raises(ValueError):
        oracle_mod.opd_kl(H_s, H_t, W_s[:, :3], W_t, mask, g, 1.0)
