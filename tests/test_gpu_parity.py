"""GPU parity: the CUDA path (through the C ABI) against the float64 CPU oracle.

Tolerances (per-token KL and gradients of the reverse KL, Section 3
Eq. reverse-kl): |KL_gpu - KL_oracle| <= 1e-4 + 2e-3 |KL_oracle| elementwise;
dH_s and dW_s within 1e-2 relative Frobenius error (bf16 inputs, fp32
accumulation, bf16 staging of dz). The float32 path is held to 1e-5 / 1e-4.

Small cases run the whole oracle; full-size workloads run the bench's launch
configuration and check a deterministic sample of rows (rows are independent
given the hidden states), plus dW_s on a mask-subsetted full-shape run.
"""

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


def _check_kl(got, want, abs_tol=KL_ABS, rel_tol=KL_REL):
    excess = np.abs(np.asarray(got, np.float64) - want) - (abs_tol + rel_tol * np.abs(want))
    assert excess.max() <= 0, f"KL worst excess {excess.max():.3e} at {int(excess.argmax())}"


def _run(lib, w, x, mask, g, *, mode="fwd_bwd", accumulate=False, dW_init=None):
    dev = x["H_s"].device
    dtype = lib.OPD_DTYPE_F32 if w.dtype == "f32" else lib.OPD_DTYPE_BF16
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, dtype, w.tau)
    ws = lib.allocate_workspace(prob, dev)
    m = torch.as_tensor(mask, device=dev, dtype=torch.uint8)
    grad = torch.as_tensor(np.asarray(g, np.float32), device=dev)
    kl = torch.full((w.T,), float("nan"), device=dev)
    stats = torch.full((w.T, 3), float("nan"), device=dev)
    dH = torch.full((w.T, w.d_s), float("nan"), device=dev)
    dW = torch.full((w.V, w.d_s), float("nan"), device=dev) if dW_init is None else dW_init.clone()
    if mode == "fwd_bwd":
        lib.opd_kl_fwd_bwd(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], m, grad, kl, stats, dH, dW, accumulate, ws)
    else:
        lib.opd_kl_forward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], m, kl, stats, ws)
        lib.opd_kl_backward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], m, stats, grad, dH, dW, accumulate, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    return {"kl": kl.cpu().numpy(), "stats": stats.cpu().numpy(), "dH": dH.cpu().numpy(), "dW": dW.cpu().numpy()}


def _host(x):
    return [synth.host_values(x[k]) for k in ("H_s", "H_t", "W_s", "W_t")]


def _g64(g, mask):
    # the GPU receives float32 weights; the oracle gets the same values widened
    return np.where(np.asarray(mask) != 0, np.asarray(g, np.float32).astype(np.float64), 0.0)


def _full_check(lib, oracle_mod, w, mask=None, g=None, tight=False, **kw):
    lay = synth.layout(w) if mask is None else None
    mask = lay.mask if mask is None else mask
    g = synth.uniform_weights(w.seed, w.T) if g is None else g
    x = synth.hidden_and_heads(w, "cuda")
    out = _run(lib, w, x, mask, g, **kw)
    ref = oracle_mod.opd_kl(*_host(x), mask, _g64(g, mask), w.tau)
    if tight:
        _check_kl(out["kl"], ref.kl, 1e-5, 1e-5)
    else:
        _check_kl(out["kl"], ref.kl)
    sup = np.asarray(mask) != 0
    assert (out["kl"][~sup] == 0).all() and (out["dH"][~sup] == 0).all()
    np.testing.assert_allclose(out["stats"][sup, 0], ref.lse_s[sup], rtol=1e-5, atol=1e-4)
    np.testing.assert_allclose(out["stats"][sup, 1], ref.lse_t[sup], rtol=1e-5, atol=1e-4)
    lim = 1e-4 if tight else GRAD_REL
    assert _rel(out["dH"], ref.dH_s) <= lim, _rel(out["dH"], ref.dH_s)
    assert _rel(out["dW"], ref.dW_s) <= lim, _rel(out["dW"], ref.dW_s)
    return out, ref, x


def test_forward_only_workspace_with_every_row_masked(lib):
    """R = 0 with the forward-only workspace, on both element types: zeros out, status OK."""
    for dtype, tdt in ((lib.OPD_DTYPE_BF16, torch.bfloat16), (lib.OPD_DTYPE_F32, torch.float32)):
        T, ds, dt, V = 300, 64, 96, 500
        prob = lib.make_problem(T, ds, dt, V, dtype, 1.0)
        ws = torch.empty(lib.opd_kl_forward_workspace_size(prob), dtype=torch.uint8, device="cuda")
        H_s, H_t = torch.ones(T, ds, dtype=tdt, device="cuda"), torch.ones(T, dt, dtype=tdt, device="cuda")
        W_s, W_t = torch.ones(V, ds, dtype=tdt, device="cuda"), torch.ones(V, dt, dtype=tdt, device="cuda")
        mask = torch.zeros(T, dtype=torch.uint8, device="cuda")
        kl = torch.full((T,), float("nan"), device="cuda")
        stats = torch.full((T, 3), float("nan"), device="cuda")
        lib.opd_kl_forward(prob, H_s, H_t, W_s, W_t, mask, kl, stats, ws)
        torch.cuda.synchronize()
        assert lib.opd_kl_get_status(ws) == lib.OPD_OK
        assert (kl == 0).all() and (stats == 0).all()


@pytest.mark.parametrize("which", ["tiny_fp32", "bf16"])
def test_forward_and_scoring_with_the_forward_only_workspace(lib, oracle_mod, which):
    """opd_kl_forward and opd_score_tokens given exactly opd_kl_forward_workspace_size bytes (no dz
    buffer) match the oracle, and write nothing past those bytes: a sentinel tail behind the
    workspace view stays intact."""
    w = synth.WORKLOADS["tiny_fp32"] if which == "tiny_fp32" else _small_bf16(T=600, seed=12)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    dtype = lib.OPD_DTYPE_F32 if w.dtype == "f32" else lib.OPD_DTYPE_BF16
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, dtype, w.tau)
    n = lib.opd_kl_forward_workspace_size(prob)
    assert 0 < n < lib.opd_kl_workspace_size(prob)
    buf = torch.full((n + 4096,), 0xA5, dtype=torch.uint8, device="cuda")
    ws = buf[:n]
    mask = torch.from_numpy(lay.mask).cuda()
    kl = torch.full((w.T,), float("nan"), device="cuda")
    stats = torch.full((w.T, 3), float("nan"), device="cuda")
    lib.opd_kl_forward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, kl, stats, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    sup = lay.mask != 0
    ref = oracle_mod.opd_kl(*_host(x), lay.mask, np.zeros(w.T), w.tau, want_dH=False, want_dW=False)
    _check_kl(kl.cpu().numpy(), ref.kl)
    st = stats.cpu().numpy()
    np.testing.assert_allclose(st[sup, 0], ref.lse_s[sup], rtol=1e-5, atol=1e-4)
    np.testing.assert_allclose(st[sup, 1], ref.lse_t[sup], rtol=1e-5, atol=1e-4)
    if dtype == lib.OPD_DTYPE_BF16:  # token scoring (bf16 only) with the same workspace
        tokens = synth.token_ids(w.seed, w.T, w.V)
        sprob = lib.make_problem(w.T, w.d_t, w.d_t, w.V, dtype, w.tau)
        m = lib.opd_kl_forward_workspace_size(sprob)
        sws = buf[:m] if m <= n else torch.empty(m, dtype=torch.uint8, device="cuda")
        lse = torch.full((w.T,), float("nan"), device="cuda")
        lp = torch.full((w.T,), float("nan"), device="cuda")
        lib.opd_score_tokens(sprob, x["H_t"], x["W_t"], torch.from_numpy(tokens).cuda(), mask, lse, lp, sws)
        torch.cuda.synchronize()
        assert lib.opd_kl_get_status(sws) == lib.OPD_OK
        ref_lse, ref_lp = oracle_mod.score(synth.host_values(x["H_t"]), synth.host_values(x["W_t"]), tokens, w.tau,
                                           rows=np.flatnonzero(sup))
        np.testing.assert_allclose(lse.cpu().numpy()[sup], ref_lse, rtol=1e-4, atol=1e-4)
        np.testing.assert_allclose(lp.cpu().numpy()[sup], ref_lp, rtol=1e-4, atol=1e-4)
    assert (buf[n:] == 0xA5).all()


@pytest.mark.parametrize("layout", ["tiny", "tiny_alt"])
def test_tiny_fp32_config(lib, oracle_mod, layout):
    w = synth.scaled(synth.WORKLOADS["tiny_fp32"], layout=layout)
    _full_check(lib, oracle_mod, w, tight=True)


def _small_bf16(**kw):
    base = dict(name="small", T=700, d_s=256, d_t=384, V=1000, tau=0.7, n_traj=7, traj_len=100, seed=11)
    base.update(kw)
    return synth.scaled(synth.WORKLOADS["qwen3_1p7b"], **base)


@pytest.fixture(params=["bn256/cta1", "pair256/cta1", "pair256/pair"])
def tiling(request, monkeypatch):
    """Tilings of the fused kernels (128 x 256 tiles on one CTA, 256 x 256 on a CTA pair) and of the
    gradient GEMMs (128 x 256 on one CTA, 256 x 256 on a pair); the library reads both overrides on
    every call."""
    fused, gemm = request.param.split("/")
    monkeypatch.setenv("OPD_KL_FUSED", fused)
    monkeypatch.setenv("OPD_KL_GEMM", gemm)
    return request.param


def test_bf16_several_tiles_ragged_vocab(lib, oracle_mod, tiling):
    # 3+ row tiles with a ragged last tile, several vocabulary tiles with a ragged tail,
    # K blocks 4 (student) and 6 (teacher)
    _full_check(lib, oracle_mod, _small_bf16())


def test_bf16_ragged_hidden_sizes_and_vocab(lib, oracle_mod, tiling):
    # d not a multiple of the 64-wide K block, d_s not a multiple of the 256-wide GEMM tile,
    # V not a multiple of 8 (dz pitch padding)
    _full_check(lib, oracle_mod, _small_bf16(T=300, d_s=200, d_t=136, V=1237, tau=1.3, n_traj=3, seed=12))


def test_bf16_many_vocab_splits(lib, oracle_mod, tiling):
    # few row tiles and a long vocabulary: the forward splits V across many CTAs
    _full_check(lib, oracle_mod, _small_bf16(T=256, d_s=64, d_t=64, V=40000, tau=1.0, n_traj=2, traj_len=128,
                                             seed=23))


@pytest.mark.parametrize("tau", [0.1, 5.0])
def test_bf16_extreme_temperatures(lib, oracle_mod, tau):
    # tau = 0.1 spreads the scaled logits over hundreds of units (one token takes nearly all
    # the mass); tau = 5 flattens both distributions
    _full_check(lib, oracle_mod, _small_bf16(T=300, V=3000, tau=tau, n_traj=3, seed=28))


def _random_cases(n, seed=2026):
    rng = np.random.default_rng(seed)
    cases = []
    for i in range(n):
        cases.append(dict(T=int(rng.integers(1, 700)), d_s=8 * int(rng.integers(1, 41)), d_t=8 * int(rng.integers(1, 49)),
                          V=int(rng.integers(2, 6000)), tau=float(rng.choice([0.3, 0.7, 1.0, 1.6])),
                          density=float(rng.uniform(0.05, 1.0)), tiling=["bn256/cta1", "pair256/pair"][i % 2],
                          seed=100 + i))
    return cases


@pytest.mark.parametrize("case", _random_cases(16), ids=lambda c: f"T{c['T']}-ds{c['d_s']}-dt{c['d_t']}-V{c['V']}")
def test_random_shapes(lib, oracle_mod, case, monkeypatch):
    """Seeded random problems: any T, hidden sizes in multiples of 8, any V, mixed temperatures and
    mask densities, on both tilings."""
    fused, gemm = case["tiling"].split("/")
    monkeypatch.setenv("OPD_KL_FUSED", fused)
    monkeypatch.setenv("OPD_KL_GEMM", gemm)
    w = _small_bf16(T=case["T"], d_s=case["d_s"], d_t=case["d_t"], V=case["V"], tau=case["tau"], n_traj=1,
                    traj_len=case["T"], seed=case["seed"])
    mask = (np.random.default_rng(case["seed"]).random(w.T) < case["density"]).astype(np.uint8)
    mask[np.random.default_rng(case["seed"] + 1).integers(0, w.T)] = 1
    _full_check(lib, oracle_mod, w, mask=mask)


@pytest.mark.parametrize("R", [1, 37, 128, 129, 293, 384])
@pytest.mark.parametrize("half", ["1", "0"])
def test_half_height_last_tile(lib, oracle_mod, monkeypatch, R, half):
    """On CTA pairs a last row tile with at most 128 supervised rows runs as M = 128 MMAs
    (64 rows per CTA; vocabulary columns 128-255 of each tile in TMEM lanes 64-127, their
    statistics a second partial per row). R = 1, 37, 128 and 293 take that path, R = 129
    and 384 do not; OPD_KL_HALF_TILE=0 runs every tile at full height. V = 4,986 leaves
    122 columns in the last vocabulary tile, so with one tile per unit the warps of
    columns 128-255 own no column there."""
    monkeypatch.setenv("OPD_KL_FUSED", "pair256")
    monkeypatch.setenv("OPD_KL_GEMM", "pair")
    monkeypatch.setenv("OPD_KL_HALF_TILE", half)
    w = _small_bf16(T=420, d_s=208, d_t=144, V=4986, tau=0.7, n_traj=1, traj_len=420, seed=31)
    mask = np.zeros(w.T, np.uint8)
    mask[np.random.default_rng(R).choice(w.T, R, replace=False)] = 1
    _full_check(lib, oracle_mod, w, mask=mask)


@pytest.mark.parametrize("env", [("OPD_KL_VSPLIT", "1"), ("OPD_KL_VSPLIT", "7"), ("OPD_KL_VSPLIT", "128"),
                                 ("OPD_KL_GROUP_ROWS", "1"), ("OPD_KL_GROUP_ROWS", "64"),
                                 ("OPD_KL_MAX_KSPLIT", "1"), ("OPD_KL_MAX_KSPLIT", "16")],
                         ids=lambda e: f"{e[0]}={e[1]}")
def test_tuning_overrides_keep_parity(lib, oracle_mod, monkeypatch, env):
    """Every schedule the tuning overrides reach computes the same result: one vocabulary split
    (a unit walks all of V), the largest split count, raster groups of one row tile or of all
    of them, and the dH_s GEMM with and without split-K. Four row-pair tiles, the last one at
    half height (R = 800)."""
    monkeypatch.setenv("OPD_KL_FUSED", "pair256")
    monkeypatch.setenv("OPD_KL_GEMM", "pair")
    monkeypatch.setenv(*env)
    w = _small_bf16(T=1000, d_s=128, d_t=192, V=3000, tau=1.0, n_traj=1, traj_len=1000, seed=37)
    mask = np.zeros(w.T, np.uint8)
    mask[np.random.default_rng(37).choice(w.T, 800, replace=False)] = 1
    _full_check(lib, oracle_mod, w, mask=mask)


def test_mask_at_any_byte_offset(lib):
    """The compaction reads the mask in 16-byte vectors when it is 16-byte aligned and byte by
    byte otherwise (a mask that is a slice of a larger one, as with row chunks): both give
    bit-identical results."""
    w = _small_bf16(T=1000, d_s=64, d_t=64, V=700, tau=1.0, n_traj=10, traj_len=100, seed=38)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob)
    outs = []
    for offset in (0, 5):
        backing = torch.zeros(w.T + 16, dtype=torch.uint8, device="cuda")
        backing[offset:offset + w.T] = torch.from_numpy(lay.mask).cuda()
        mask = backing[offset:offset + w.T]
        assert (mask.data_ptr() % 16 == 0) == (offset == 0)
        kl = torch.full((w.T,), float("nan"), device="cuda")
        st = torch.full((w.T, 3), float("nan"), device="cuda")
        lib.opd_kl_forward(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, kl, st, ws)
        torch.cuda.synchronize()
        assert lib.opd_kl_get_status(ws) == lib.OPD_OK
        outs.append((kl.cpu().numpy(), st.cpu().numpy()))
    np.testing.assert_array_equal(outs[0][0], outs[1][0])
    np.testing.assert_array_equal(outs[0][1], outs[1][1])
    sup = lay.mask != 0
    assert (outs[0][0][~sup] == 0).all() and (outs[0][0][sup] > 0).all()


def test_bf16_correlated_teacher_small_kl(lib, oracle_mod):
    w = _small_bf16(T=256, d_s=128, d_t=320, V=2048, tau=1.0, n_traj=2, traj_len=128, correlated_teacher=True,
                    seed=13)
    out, ref, _ = _full_check(lib, oracle_mod, w)
    sup = synth.layout(w).mask != 0
    assert np.median(ref.kl[sup]) < 1.0


def test_forward_then_backward_matches_fused_call(lib):
    w = _small_bf16(T=400, seed=14)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    a = _run(lib, w, x, lay.mask, g, mode="fwd_bwd")
    b = _run(lib, w, x, lay.mask, g, mode="separate")
    np.testing.assert_array_equal(a["kl"], b["kl"])
    np.testing.assert_array_equal(a["stats"], b["stats"])
    assert _rel(b["dH"], a["dH"].astype(np.float64)) < 1e-5
    assert _rel(b["dW"], a["dW"].astype(np.float64)) < 1e-5


def test_repeated_calls_are_deterministic(lib):
    """The forward writes each split's partial statistics once and combines them in a fixed
    order, and dW_s tiles are stored (K = R whole per tile), so KL, stats and dW_s repeat bit for
    bit. dH_s sums split-K partials by reduce-adds in arrival order: equal to rounding."""
    w = _small_bf16(T=600, V=3000, seed=29)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    a = _run(lib, w, x, lay.mask, g)
    b = _run(lib, w, x, lay.mask, g)
    np.testing.assert_array_equal(a["kl"], b["kl"])
    np.testing.assert_array_equal(a["stats"], b["stats"])
    np.testing.assert_array_equal(a["dW"], b["dW"])
    assert _rel(a["dH"], b["dH"].astype(np.float64)) < 1e-6


def test_deterministic_mode(lib, oracle_mod, monkeypatch):
    """OPD_KL_DETERMINISTIC=1: dH_s tiles take the whole K range and are stored, so every output
    repeats bit for bit, and the results still match the oracle."""
    monkeypatch.setenv("OPD_KL_DETERMINISTIC", "1")
    w = _small_bf16(T=600, V=3000, seed=30)
    a, _, x = _full_check(lib, oracle_mod, w)
    lay = synth.layout(w)
    b = _run(lib, w, x, lay.mask, synth.uniform_weights(w.seed, w.T))
    for k in ("kl", "stats", "dH", "dW"):
        np.testing.assert_array_equal(a[k], b[k])


def test_row_chunks_with_accumulate_equal_one_call(lib):
    """A batch split into row chunks (per-token upstream weights computed once for the whole
    batch, one call per chunk, dW_s accumulated after the first) reproduces the single call: the
    way to bound the workspace (its dz buffer grows as T x V)."""
    w = _small_bf16(T=900, V=2000, seed=31)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    whole = _run(lib, w, x, lay.mask, g)
    cuts = [0, 300, 650, 900]
    dW = torch.zeros(w.V, w.d_s, device="cuda")
    kl, dH = np.zeros(w.T, np.float32), np.zeros((w.T, w.d_s), np.float32)
    for i, (a, b) in enumerate(zip(cuts[:-1], cuts[1:])):
        wc = synth.scaled(w, T=b - a)
        xc = {"H_s": x["H_s"][a:b], "H_t": x["H_t"][a:b], "W_s": x["W_s"], "W_t": x["W_t"]}
        out = _run(lib, wc, xc, lay.mask[a:b], g[a:b], accumulate=i > 0, dW_init=dW)
        dW = torch.from_numpy(out["dW"]).cuda()
        kl[a:b], dH[a:b] = out["kl"], out["dH"]
    np.testing.assert_array_equal(kl, whole["kl"])
    assert _rel(dH, whole["dH"].astype(np.float64)) < 1e-5
    assert _rel(dW.cpu().numpy(), whole["dW"].astype(np.float64)) < 1e-5


def test_accumulate_dW_adds(lib):
    w = _small_bf16(T=300, seed=15)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    plain = _run(lib, w, x, lay.mask, g)
    init = torch.randn(w.V, w.d_s, device="cuda", generator=torch.Generator("cuda").manual_seed(0))
    acc = _run(lib, w, x, lay.mask, g, accumulate=True, dW_init=init)
    assert _rel(acc["dW"] - init.cpu().numpy(), plain["dW"].astype(np.float64)) < 1e-5


def test_all_rows_masked(lib):
    w = _small_bf16(T=200, seed=16)
    mask = np.zeros(w.T, np.uint8)
    x = synth.hidden_and_heads(w, "cuda")
    out = _run(lib, w, x, mask, np.ones(w.T))
    assert (out["kl"] == 0).all() and (out["dH"] == 0).all() and (out["dW"] == 0).all()
    init = torch.ones(w.V, w.d_s, device="cuda")
    acc = _run(lib, w, x, mask, np.ones(w.T), accumulate=True, dW_init=init)
    assert (acc["dW"] == 1).all()


@pytest.mark.parametrize("rows", [[0], [199], [5, 6, 7, 127, 128, 129]])
def test_few_supervised_rows(lib, oracle_mod, rows, tiling):
    w = _small_bf16(T=200, seed=17)
    mask = np.zeros(w.T, np.uint8)
    mask[rows] = 1
    _full_check(lib, oracle_mod, w, mask=mask)


@pytest.mark.parametrize("shape", [
    dict(T=40, d_s=8, d_t=16, V=2),     # two-token vocabulary, hidden sizes far below one K block
    dict(T=100, d_s=16, d_t=8, V=64),   # the whole vocabulary inside a quarter of one tile
    dict(T=1, d_s=64, d_t=128, V=300),  # a single token
])
def test_shapes_below_one_tile(lib, oracle_mod, shape, tiling):
    w = _small_bf16(n_traj=1, traj_len=shape["T"], seed=21, **shape)
    mask = (np.arange(w.T) % 3 != 1).astype(np.uint8)
    mask[0] = 1
    _full_check(lib, oracle_mod, w, mask=mask)


@pytest.mark.parametrize("case", range(4))
def test_fp32_random_shapes(lib, oracle_mod, case):
    """The CUDA-core float32 path on seeded random small problems (any hidden size), tight bounds."""
    rng = np.random.default_rng(300 + case)
    w = synth.scaled(synth.WORKLOADS["tiny_fp32"], T=int(rng.integers(1, 120)), d_s=int(rng.integers(1, 96)),
                     d_t=int(rng.integers(1, 160)), V=int(rng.integers(2, 1500)), tau=float(rng.uniform(0.5, 2.0)),
                     seed=300 + case)
    mask = (rng.random(w.T) < 0.7).astype(np.uint8)
    mask[0] = 1
    _full_check(lib, oracle_mod, w, mask=mask, tight=True)


def test_fp32_two_token_vocabulary(lib, oracle_mod):
    w = synth.scaled(synth.WORKLOADS["tiny_fp32"], V=2, d_s=8, d_t=16, seed=22)
    _full_check(lib, oracle_mod, w, tight=True)


def test_cuda_graph_capture_and_replay(lib, oracle_mod):
    """The ABI never synchronises the host, so a whole step can be captured in a CUDA graph;
    replays give the eager call's results on the same inputs, and on new inputs copied into the
    captured buffers."""
    w = _small_bf16(T=400, seed=24)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    eager = _run(lib, w, x, lay.mask, g)

    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    ws = lib.allocate_workspace(prob, "cuda")
    m = torch.as_tensor(lay.mask, device="cuda", dtype=torch.uint8)
    grad = torch.as_tensor(np.asarray(g, np.float32), device="cuda")
    H_s, H_t = x["H_s"].clone(), x["H_t"].clone()
    kl = torch.empty(w.T, device="cuda")
    stats = torch.empty(w.T, 3, device="cuda")
    dH = torch.empty(w.T, w.d_s, device="cuda")
    dW = torch.empty(w.V, w.d_s, device="cuda")

    def step():
        lib.opd_kl_fwd_bwd(prob, H_s, H_t, x["W_s"], x["W_t"], m, grad, kl, stats, dH, dW, False, ws)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()  # first call outside the capture: kernel attributes are set here
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    for t in (kl, stats, dH, dW):
        t.fill_(float("nan"))
    graph.replay()
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    np.testing.assert_array_equal(kl.cpu().numpy(), eager["kl"])
    assert _rel(dH.cpu().numpy(), eager["dH"].astype(np.float64)) < 1e-5
    assert _rel(dW.cpu().numpy(), eager["dW"].astype(np.float64)) < 1e-5

    # new hidden states through the same graph: checked against the oracle
    x2 = synth.hidden_and_heads(synth.scaled(w, seed=25), "cuda")
    H_s.copy_(x2["H_s"])
    H_t.copy_(x2["H_t"])
    graph.replay()
    torch.cuda.synchronize()
    ref = oracle_mod.opd_kl(synth.host_values(x2["H_s"]), synth.host_values(x2["H_t"]),
                            synth.host_values(x["W_s"]), synth.host_values(x["W_t"]), lay.mask,
                            _g64(g, lay.mask), w.tau)
    _check_kl(kl.cpu().numpy(), ref.kl)
    assert _rel(dH.cpu().numpy(), ref.dH_s) <= GRAD_REL
    assert _rel(dW.cpu().numpy(), ref.dW_s) <= GRAD_REL


def test_debug_mode_reports_non_finite_outputs(lib, monkeypatch):
    """With OPD_KL_SYNC_CHECK=1 every call scans its outputs: a NaN in one supervised hidden row
    comes back as OPD_ERR_NONFINITE. Without it nothing is checked (inputs must be finite)."""
    w = _small_bf16(T=128, d_s=64, d_t=64, V=300, n_traj=1, traj_len=128, seed=26)
    x = synth.hidden_and_heads(w, "cuda")
    mask = np.ones(w.T, np.uint8)
    monkeypatch.setenv("OPD_KL_SYNC_CHECK", "1")
    clean = _run(lib, w, x, mask, np.ones(w.T))
    assert np.isfinite(clean["kl"]).all()
    x["H_s"] = x["H_s"].clone()
    x["H_s"][5, 3] = float("nan")
    with pytest.raises(lib.OpdError) as err:
        _run(lib, w, x, mask, np.ones(w.T))
    assert err.value.status == lib.OPD_ERR_NONFINITE
    monkeypatch.delenv("OPD_KL_SYNC_CHECK")
    out = _run(lib, w, x, mask, np.ones(w.T))
    assert np.isnan(out["kl"][5]) and np.isfinite(np.delete(out["kl"], 5)).all()


def test_empty_batch(lib):
    """T = 0: every call succeeds; dW_s is zeroed, or left untouched when accumulating."""
    d_s, d_t, V = 64, 128, 300
    prob = lib.make_problem(0, d_s, d_t, V, lib.OPD_DTYPE_BF16, 1.0)
    ws = lib.allocate_workspace(prob, "cuda")
    e = lambda *shape, dt=torch.bfloat16: torch.empty(*shape, device="cuda", dtype=dt)
    W_s, W_t = torch.randn(V, d_s, device="cuda").bfloat16(), torch.randn(V, d_t, device="cuda").bfloat16()
    f32 = lambda *shape: torch.empty(*shape, device="cuda")
    dW = torch.full((V, d_s), float("nan"), device="cuda")
    lib.opd_kl_fwd_bwd(prob, e(0, d_s), e(0, d_t), W_s, W_t, e(0, dt=torch.uint8), f32(0), f32(0), f32(0, 3),
                       f32(0, d_s), dW, False, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    assert (dW == 0).all()
    dW.fill_(2.0)
    lib.opd_kl_fwd_bwd(prob, e(0, d_s), e(0, d_t), W_s, W_t, e(0, dt=torch.uint8), f32(0), f32(0), f32(0, 3),
                       f32(0, d_s), dW, True, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    assert (dW == 2.0).all()
    prob1 = lib.make_problem(0, d_s, d_s, V, lib.OPD_DTYPE_BF16, 1.0)
    tok = torch.empty(0, device="cuda", dtype=torch.int32)
    lib.opd_score_tokens(prob1, e(0, d_s), W_s, tok, e(0, dt=torch.uint8), f32(0), f32(0), ws)
    dW.fill_(float("nan"))
    lib.opd_surrogate_fwd_bwd(prob1, e(0, d_s), W_s, tok, f32(0), f32(0), e(0, dt=torch.uint8), f32(0), f32(0),
                              f32(0), f32(0, d_s), dW, False, ws)
    torch.cuda.synchronize()
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK
    assert (dW == 0).all()


def test_student_equals_teacher_gives_zero(lib):
    w = _small_bf16(T=256, d_t=256, seed=18)
    lay = synth.layout(w)
    x = synth.hidden_and_heads(w, "cuda")
    x["H_t"], x["W_t"] = x["H_s"], x["W_s"]
    out = _run(lib, w, x, lay.mask, synth.uniform_weights(w.seed, w.T))
    assert np.abs(out["kl"]).max() < 2e-5
    # dz = p_s (log p_s - log p_t - KL) vanishes up to fp32 rounding of identical logits
    assert np.abs(out["dH"]).max() < 1e-4 and np.abs(out["dW"]).max() < 1e-4


def test_bounded_wait_timeout_reports_and_context_survives(lib):
    prob = lib.make_problem(64, 64, 64, 64, lib.OPD_DTYPE_BF16, 1.0)
    ws = lib.allocate_workspace(prob)
    assert lib.opd_kl_selftest_timeout(ws, 50_000_000) == lib.OPD_ERR_TIMEOUT
    assert lib.opd_kl_get_status(ws) == lib.OPD_OK  # status was cleared
    w = _small_bf16(T=128, d_s=64, d_t=64, V=64, n_traj=1, traj_len=128, seed=19)
    x = synth.hidden_and_heads(w, "cuda")
    out = _run(lib, w, x, synth.layout(w).mask, np.ones(w.T))
    assert np.isfinite(out["kl"]).all()


FULL = ["qwen3_0p6b", "qwen3_1p7b", "qwen3_4b", "ragged_multiturn"]


def test_largest_batch_sampled_rows(lib, oracle_mod):
    """T = 131,072 packed tokens (twice the ragged workload): dz alone is 40 GB, so byte offsets
    pass 2^32; sampled rows against the oracle, which gets only those rows (rows are independent)."""
    w = synth.scaled(synth.WORKLOADS["qwen3_1p7b"], name="largest", T=131072, n_traj=256, seed=27)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    out = _run(lib, w, x, lay.mask, g)
    sup = lay.mask != 0
    assert (out["kl"][~sup] == 0).all() and (out["dH"][~sup] == 0).all() and np.isfinite(out["dW"]).all()
    rows = np.flatnonzero(sup)
    pick = np.unique(np.concatenate([rows[np.linspace(0, len(rows) - 1, 12).astype(int)], rows[-2:]]))
    sel = torch.as_tensor(pick, device="cuda")
    H_s, H_t = (synth.host_values(x[k].index_select(0, sel)) for k in ("H_s", "H_t"))
    W_s, W_t = synth.host_values(x["W_s"]), synth.host_values(x["W_t"])
    ones = np.ones(len(pick), np.uint8)
    ref = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, ones, _g64(g[pick], ones), w.tau)
    _check_kl(out["kl"][pick], ref.kl)
    assert _rel(out["dH"][pick], ref.dH_s) <= GRAD_REL
    # dW_s at the same size with only the sampled rows supervised
    mask2 = np.zeros_like(lay.mask)
    mask2[pick] = 1
    out2 = _run(lib, w, x, mask2, g)
    assert _rel(out2["dW"], ref.dW_s) <= GRAD_REL, _rel(out2["dW"], ref.dW_s)


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled_rows(lib, oracle_mod, name):
    w = synth.WORKLOADS[name]
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    out = _run(lib, w, x, lay.mask, g)
    sup = lay.mask != 0
    # properties at any size
    assert (out["kl"][~sup] == 0).all() and (out["dH"][~sup] == 0).all()
    assert out["kl"][sup].min() > -1e-4 and np.isfinite(out["dW"]).all()
    # sampled rows against the oracle
    rows = np.flatnonzero(sup)
    pick = np.unique(np.concatenate([rows[np.linspace(0, len(rows) - 1, 16).astype(int)], rows[:2], rows[-2:]]))
    H_s, H_t, W_s, W_t = _host(x)
    ref = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, lay.mask, _g64(g, lay.mask), w.tau, rows=pick, want_dW=False)
    _check_kl(out["kl"][pick], ref.kl)
    assert _rel(out["dH"][pick], ref.dH_s) <= GRAD_REL
    # dW_s on the same shapes with only a few supervised rows
    sub = pick[::2]
    mask2 = np.zeros_like(lay.mask)
    mask2[sub] = 1
    out2 = _run(lib, w, x, mask2, g)
    ref2 = oracle_mod.opd_kl(H_s, H_t, W_s, W_t, mask2, _g64(g, mask2), w.tau, rows=sub, want_dH=False)
    assert _rel(out2["dW"], ref2.dW_s) <= GRAD_REL, _rel(out2["dW"], ref2.dW_s)
    _check_kl(out2["kl"][sub], ref2.kl)


def test_row_chunk_helper_under_a_workspace_budget(lib, oracle_mod):
    """kl_fwd_bwd_in_row_chunks with a budget that holds 256 rows: four chunks of one shared
    workspace, against one call and against the oracle; with accumulate_dW the first chunk adds
    to dW_s too."""
    from paper_2609_36608_gb300 import chunking
    w = _small_bf16(T=900, V=2000, seed=32)
    lay = synth.layout(w)
    g = synth.uniform_weights(w.seed, w.T)
    x = synth.hidden_and_heads(w, "cuda")
    whole = _run(lib, w, x, lay.mask, g)
    prob = lib.make_problem(w.T, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau)
    budget = lib.opd_kl_workspace_size(lib.make_problem(256, w.d_s, w.d_t, w.V, lib.OPD_DTYPE_BF16, w.tau))
    assert chunking.max_rows_for_workspace(prob, budget) == 256
    mask = torch.from_numpy(lay.mask).cuda()
    grad = torch.from_numpy(np.asarray(g, np.float32)).cuda()
    kl, stats = torch.full((w.T,), float("nan"), device="cuda"), torch.full((w.T, 3), float("nan"), device="cuda")
    dH = torch.full((w.T, w.d_s), float("nan"), device="cuda")
    init = torch.randn(w.V, w.d_s, device="cuda", generator=torch.Generator("cuda").manual_seed(3))
    dW = init.clone()
    n = chunking.kl_fwd_bwd_in_row_chunks(prob, x["H_s"], x["H_t"], x["W_s"], x["W_t"], mask, grad, kl, stats, dH,
                                          dW, True, budget)
    torch.cuda.synchronize()
    assert n == 4
    got_kl = kl.cpu().numpy()
    np.testing.assert_allclose(got_kl, whole["kl"], rtol=1e-6, atol=1e-7)
    assert _rel(dH.cpu().numpy(), whole["dH"].astype(np.float64)) < 1e-5
    assert _rel((dW - init).cpu().numpy(), whole["dW"].astype(np.float64)) < 1e-5
    ref = oracle_mod.opd_kl(*_host(x), lay.mask, _g64(g, lay.mask), w.tau)
    _check_kl(got_kl, ref.kl)
    assert _rel(dH.cpu().numpy(), ref.dH_s) <= GRAD_REL
    assert _rel((dW - init).cpu().numpy(), ref.dW_s) <= GRAD_REL
