"""Pins for the oracle's token scoring and sampled-token surrogate (Appendix B.4).

Each fact below is independent of the oracle's own code:

- a hand-worked table of the piecewise dual-clip loss and its slope, one row per branch
  (tests/golden/dual_clip.txt);
- the on-policy case rho = 1, where the surrogate reduces to the policy gradient
  -A (1[k = x] - p) / tau, checked against scipy's softmax;
- zero-sum gradient rows;
- inert masked rows;
- finite differences of the weighted loss, with inputs kept away from the kinks;
- a float64 PyTorch autograd evaluation of the same loss;
- scoring against scipy's logsumexp and the reverse-KL oracle's log-partition values.
"""

import math
import os

import numpy as np
import pytest
import scipy.special as sp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _head(seed, T=9, d=6, V=31, std=2.0):
    rng = np.random.default_rng(seed)
    H = rng.standard_normal((T, d)).astype(np.float32)
    W = (rng.standard_normal((V, d)) * std / math.sqrt(d)).astype(np.float32)
    tokens = rng.integers(0, V, T).astype(np.int32)
    return H, W, tokens


def _away_from_kinks(oracle_mod, H, W, tokens, tau, seed, mask):
    """logp_old and logp_teacher whose ratio and advantage keep every token at least 0.02 (in
    log-ratio) away from the clip boundaries 1 +- 0.2 and the dual-clip threshold rho = 3."""
    rng = np.random.default_rng(seed)
    _, lp = oracle_mod.score(H, W, tokens, tau)
    T = len(tokens)
    r = np.empty(T)
    edges = np.log([0.8, 1.2, 3.0])
    for i in range(T):
        while True:
            x = rng.uniform(-0.6, 1.4)
            if np.min(np.abs(x - edges)) > 0.02:
                r[i] = x
                break
    logp_old = lp - r
    A = rng.choice([-1.0, 1.0], T) * rng.uniform(0.2, 1.5, T)
    logp_teacher = logp_old + A
    w = rng.uniform(0.5, 1.5, T) * (np.asarray(mask) != 0)
    return logp_old, logp_teacher, w


def test_dual_clip_hand_table(oracle_mod):
    rows = []
    with open(os.path.join(GOLDEN, "dual_clip.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    logp_s = []
    for r in rows:
        logp_s.append(25.0 if r[0] == "inf+" else (-25.0 if r[0] == "inf-" else math.log(float(r[0]))))
    A = [float(r[1]) for r in rows]
    want_loss = np.array([float(r[2]) for r in rows])
    want_slope = np.array([float(r[3]) for r in rows])
    loss, slope = oracle_mod.dual_clip(np.array(logp_s), np.zeros(len(rows)), np.array(A))
    np.testing.assert_allclose(loss, want_loss, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(slope, want_slope, rtol=1e-12, atol=1e-15)


def test_score_matches_scipy_and_kl_oracle(oracle_mod):
    H, W, tokens = _head(1)
    tau = 0.7
    lse, lp = oracle_mod.score(H, W, tokens, tau)
    u = (H.astype(np.float64) @ W.astype(np.float64).T) / tau
    np.testing.assert_allclose(lse, sp.logsumexp(u, axis=1), rtol=1e-13)
    np.testing.assert_allclose(lp, u[np.arange(len(tokens)), tokens] - sp.logsumexp(u, axis=1), rtol=1e-12,
                               atol=1e-13)
    # the same log-partition through the reverse-KL oracle's student side
    kl = oracle_mod.opd_kl(H, H, W, W, np.ones(len(tokens), np.uint8), np.ones(len(tokens)), tau,
                           want_dH=False, want_dW=False)
    np.testing.assert_allclose(lse, kl.lse_s, rtol=1e-14)


def test_score_hand_three_token_example(oracle_mod):
    # student logits (0, ln 2, 0): p = (1/4, 1/2, 1/4), lse = ln 4; token 1 -> log p = ln(1/2)
    ln2 = np.float32(math.log(2.0))
    H = np.ones((2, 1), np.float32)
    W = np.array([[0.0], [ln2], [0.0]], np.float32)
    lse, lp = oracle_mod.score(H, W, np.array([1, 2], np.int32))
    assert abs(lse[0] - math.log(4.0)) < 1e-7
    assert abs(lp[0] - math.log(0.5)) < 1e-7 and abs(lp[1] - math.log(0.25)) < 1e-7


def test_on_policy_surrogate_is_the_policy_gradient(oracle_mod):
    H, W, tokens = _head(2)
    tau = 1.3
    T = len(tokens)
    _, lp = oracle_mod.score(H, W, tokens, tau)
    rng = np.random.default_rng(0)
    A = rng.uniform(-1.5, 1.5, T)
    w = rng.uniform(0.5, 1.5, T)
    mask = np.ones(T, np.uint8)
    res = oracle_mod.surrogate(H, W, tokens, lp, lp + A, mask, w, tau, want_dZ=True)
    # rho = 1: l = -A (clip and dual clip inactive), d l / d logp = -A
    np.testing.assert_allclose(res.loss, -A, rtol=1e-12, atol=1e-14)
    p = sp.softmax((H.astype(np.float64) @ W.astype(np.float64).T) / tau, axis=1)
    onehot = np.zeros_like(p)
    onehot[np.arange(T), tokens] = 1.0
    dz = (-A * w / tau)[:, None] * (onehot - p)
    np.testing.assert_allclose(res.dZ, dz, rtol=1e-10, atol=1e-15)


def test_surrogate_gradient_rows_sum_to_zero_and_masking(oracle_mod):
    H, W, tokens = _head(3, T=12)
    mask = np.array([1, 0, 1, 1, 0, 1, 1, 1, 0, 1, 1, 1], np.uint8)
    lo, lt, w = _away_from_kinks(oracle_mod, H, W, tokens, 1.0, 5, mask)
    res = oracle_mod.surrogate(H, W, tokens, lo, lt, mask, w, 1.0, want_dZ=True)
    scale = np.abs(res.dZ).sum(axis=1)
    assert (np.abs(res.dZ.sum(axis=1)) <= 1e-14 * np.maximum(scale, 1.0)).all()
    assert (res.loss[mask == 0] == 0).all() and (res.dZ[mask == 0] == 0).all()
    H2 = H.copy()
    H2[mask == 0] *= -3.0
    lo2 = lo.copy()
    lo2[mask == 0] += 5.0
    res2 = oracle_mod.surrogate(H2, W, tokens, lo2, lt, mask, w, 1.0)
    np.testing.assert_array_equal(res2.dW_s, res.dW_s)
    np.testing.assert_array_equal(res2.loss[mask == 1], res.loss[mask == 1])


@pytest.mark.parametrize("tau", [1.0, 0.7])
def test_surrogate_finite_differences(oracle_mod, tau):
    H, W, tokens = _head(4, T=6, d=4, V=11)
    mask = np.ones(6, np.uint8)
    lo, lt, w = _away_from_kinks(oracle_mod, H, W, tokens, tau, 6, mask)
    res = oracle_mod.surrogate(H, W, tokens, lo, lt, mask, w, tau)

    def L(Hx, Wx):
        r = oracle_mod.surrogate(Hx, Wx, tokens, lo, lt, mask, w, tau, want_dH=False, want_dW=False)
        return float(np.dot(w, r.loss))

    h = 2.0 ** -12
    rng = np.random.default_rng(7)
    for _ in range(10):
        i, j = rng.integers(0, 6), rng.integers(0, 4)
        Hp, Hm = H.copy(), H.copy()
        Hp[i, j] += np.float32(h)
        Hm[i, j] -= np.float32(h)
        fd = (L(Hp, W) - L(Hm, W)) / (float(Hp[i, j]) - float(Hm[i, j]))
        assert abs(fd - res.dH_s[i, j]) <= 1e-5 * max(1.0, abs(fd)), (i, j, fd, res.dH_s[i, j])
        k, j = rng.integers(0, 11), rng.integers(0, 4)
        Wp, Wm = W.copy(), W.copy()
        Wp[k, j] += np.float32(h)
        Wm[k, j] -= np.float32(h)
        fd = (L(H, Wp) - L(H, Wm)) / (float(Wp[k, j]) - float(Wm[k, j]))
        assert abs(fd - res.dW_s[k, j]) <= 1e-5 * max(1.0, abs(fd)), (k, j, fd, res.dW_s[k, j])


def test_surrogate_torch_autograd_cross_check(oracle_mod):
    torch = pytest.importorskip("torch")
    H, W, tokens = _head(5, T=14, d=8, V=40)
    tau = 0.8
    mask = (np.arange(14) % 5 != 0).astype(np.uint8)
    lo, lt, w = _away_from_kinks(oracle_mod, H, W, tokens, tau, 8, mask)
    res = oracle_mod.surrogate(H, W, tokens, lo, lt, mask, w, tau)
    h = torch.tensor(H, dtype=torch.float64, requires_grad=True)
    wt = torch.tensor(W, dtype=torch.float64, requires_grad=True)
    lp = torch.log_softmax(h @ wt.T / tau, dim=-1).gather(1, torch.tensor(tokens, dtype=torch.int64)[:, None])[:, 0]
    m = torch.tensor(mask, dtype=torch.float64)
    A = (torch.tensor(lt) - torch.tensor(lo)) * m
    rho = torch.exp(torch.clamp(lp - torch.tensor(lo), -20.0, 20.0))
    l_clip = -torch.minimum(rho * A, torch.clamp(rho, 0.8, 1.2) * A)
    l = torch.where(A < 0, torch.minimum(l_clip, -3.0 * A), l_clip) * m
    (l * torch.tensor(w)).sum().backward()
    np.testing.assert_allclose(res.loss, l.detach().numpy(), rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(res.dH_s, h.grad.numpy(), rtol=1e-9, atol=1e-13)
    np.testing.assert_allclose(res.dW_s, wt.grad.numpy(), rtol=1e-9, atol=1e-13)
