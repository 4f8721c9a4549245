"""Host-side checks of the C ABI that need no GPU: the library loads, exports
every entry point include/opd_kl.h declares, validates arguments before any
CUDA call, sizes the workspace, and its seq-mean-token-mean helper agrees with
the oracle (Appendix B.4, Eq. opd-surrogate)."""

import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_36608_gb300 import build
    build.build()
    from paper_2609_36608_gb300 import opd_kl
    return opd_kl


def _declared_functions():
    text = open(os.path.join(ROOT, "include", "opd_kl.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\*?\s*(opd_[a-z0-9_]+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(lib):
    names = _declared_functions()
    assert "opd_kl_forward" in names and "opd_kl_backward" in names and len(names) >= 8
    so = ctypes.CDLL(lib.LIBRARY_PATH)
    for n in names:
        assert hasattr(so, n), n


def test_status_strings(lib):
    assert lib.opd_status_string(0) == "OPD_OK"
    assert lib.opd_status_string(4) == "OPD_ERR_TIMEOUT"
    assert lib.opd_status_string(99) == "OPD_ERR_UNKNOWN"


def test_workspace_size(lib):
    p = lib.make_problem(16384, 2048, 4096, 151936, lib.OPD_DTYPE_BF16, 1.0)
    n = lib.opd_kl_workspace_size(p)
    # dominated by the bf16 dz buffer of T x round_up(V, 64) elements
    assert n >= 16384 * 151936 * 2 and n < 16384 * 151936 * 2 * 1.2
    assert lib.opd_kl_workspace_size(lib.make_problem(64, 64, 128, 1000, lib.OPD_DTYPE_F32, 1.0)) > 64 * 1000 * 4
    for bad in (lib.make_problem(-1, 8, 8, 8), lib.make_problem(8, 0, 8, 8), lib.make_problem(8, 8, 8, 0),
                lib.make_problem(8, 8, 8, 8, 7), lib.make_problem(8, 8, 8, 8, 0, 0.0),
                lib.make_problem(8, 8, 8, 8, 0, float("nan")), lib.make_problem(8, 12, 8, 8, 0)):
        assert lib.opd_kl_workspace_size(bad) == 0


def test_forward_workspace_is_the_leading_part_without_dz(lib):
    for T, ds, dt, V, dtype in ((16384, 2048, 4096, 151936, lib.OPD_DTYPE_BF16), (300, 64, 128, 1000, lib.OPD_DTYPE_BF16),
                                (64, 64, 128, 1000, lib.OPD_DTYPE_F32)):
        p = lib.make_problem(T, ds, dt, V, dtype, 1.0)
        full, fwd = lib.opd_kl_workspace_size(p), lib.opd_kl_forward_workspace_size(p)
        elem = 2 if dtype == lib.OPD_DTYPE_BF16 else 4
        assert 0 < fwd and fwd + T * V * elem <= full  # no dz buffer in the forward's part
        assert fwd % 256 == 0
    p = lib.make_problem(16384, 2048, 4096, 151936, lib.OPD_DTYPE_BF16, 1.0)
    assert lib.opd_kl_forward_workspace_size(p) < 0.25e9  # the gathered rows and statistics
    assert lib.opd_kl_forward_workspace_size(lib.make_problem(8, 12, 8, 8)) == 0
    # forward-only calls accept the smaller workspace (the call then stops at the missing GPU, or
    # runs); one byte less, and any backward with it, are rejected before any CUDA call
    vp = ctypes.c_void_p
    fake = vp(1 << 20)
    small = lib.make_problem(300, 64, 128, 1000, lib.OPD_DTYPE_BF16, 1.0)
    n = lib.opd_kl_forward_workspace_size(small)
    fwd = lambda nbytes: lib.call_raw("opd_kl_forward", ctypes.byref(small), fake, fake, fake, fake, fake, fake,
                                      fake, fake, ctypes.c_size_t(nbytes), None)
    assert fwd(n - 1) == lib.OPD_ERR_INVALID_ARG
    assert fwd(n) != lib.OPD_ERR_INVALID_ARG
    score = lambda nbytes: lib.call_raw("opd_score_tokens", ctypes.byref(small), fake, fake, fake, fake, fake,
                                        fake, fake, ctypes.c_size_t(nbytes), None)
    assert score(n - 1) == lib.OPD_ERR_INVALID_ARG
    assert score(n) != lib.OPD_ERR_INVALID_ARG
    rc = lib.call_raw("opd_kl_backward", ctypes.byref(small), fake, fake, fake, fake, fake, fake, fake, fake, fake,
                      0, fake, ctypes.c_size_t(n), None)
    assert rc == lib.OPD_ERR_INVALID_ARG


def test_invalid_arguments_rejected_before_any_launch(lib):
    vp = ctypes.c_void_p
    fake = vp(1 << 20)  # never dereferenced: validation fails first
    bad = lib.make_problem(8, 8, 8, 8, lib.OPD_DTYPE_BF16, -1.0)
    rc = lib.call_raw("opd_kl_forward", ctypes.byref(bad), fake, fake, fake, fake, fake, fake, fake, fake,
                      ctypes.c_size_t(1 << 20), None)
    assert rc == lib.OPD_ERR_INVALID_ARG
    odd = lib.make_problem(8, 12, 8, 8, lib.OPD_DTYPE_BF16, 1.0)
    rc = lib.call_raw("opd_kl_forward", ctypes.byref(odd), fake, fake, fake, fake, fake, fake, fake, fake,
                      ctypes.c_size_t(1 << 20), None)
    assert rc == lib.OPD_ERR_UNSUPPORTED
    ok = lib.make_problem(8, 8, 8, 8, lib.OPD_DTYPE_BF16, 1.0)
    rc = lib.call_raw("opd_kl_forward", ctypes.byref(ok), fake, fake, fake, fake, fake, fake, fake, None,
                      ctypes.c_size_t(0), None)
    assert rc == lib.OPD_ERR_INVALID_ARG  # no workspace
    rc = lib.call_raw("opd_kl_forward", ctypes.byref(ok), fake, fake, fake, fake, fake, fake, fake, vp(4096 + 8),
                      ctypes.c_size_t(1 << 20), None)
    assert rc == lib.OPD_ERR_INVALID_ARG  # misaligned workspace
    rc = lib.call_raw("opd_kl_forward", None, fake, fake, fake, fake, fake, fake, fake, fake,
                      ctypes.c_size_t(1 << 20), None)
    assert rc == lib.OPD_ERR_INVALID_ARG
    rc = lib.call_raw("opd_kl_selftest_timeout", fake, ctypes.c_size_t(1 << 20), ctypes.c_uint64(0), None)
    assert rc == lib.OPD_ERR_INVALID_ARG


def test_seq_mean_token_mean_helper_matches_oracle(lib, oracle_mod):
    from paper_2609_36608_gb300 import synth
    for name in ("tiny_fp32", "qwen3_0p6b", "ragged_multiturn"):
        lay = synth.layout(synth.WORKLOADS[name])
        w = lib.opd_seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
        ref = oracle_mod.seq_mean_token_mean_weights(lay.seg_id, lay.mask, 1e-8)
        np.testing.assert_allclose(w, ref, rtol=2e-7, atol=0)
    with pytest.raises(lib.OpdError):
        lib.opd_seq_mean_token_mean_weights(np.zeros(3, np.int32), np.zeros(3, np.uint8), -1.0)


def test_seq_mean_token_mean_device_arguments(lib):
    assert lib.opd_seq_mean_token_mean_workspace_size(0) == 0
    assert lib.opd_seq_mean_token_mean_workspace_size(100) >= 256 + 16 + 800
    vp = ctypes.c_void_p
    fake = vp(1 << 20)
    # no output requested
    rc = lib.call_raw("opd_seq_mean_token_mean_device", fake, fake, ctypes.c_int64(4), ctypes.c_int64(2),
                      ctypes.c_float(1e-8), None, None, None, fake, ctypes.c_size_t(4096), None)
    assert rc == lib.OPD_ERR_INVALID_ARG
    # workspace too small
    rc = lib.call_raw("opd_seq_mean_token_mean_device", fake, fake, ctypes.c_int64(4), ctypes.c_int64(1000),
                      ctypes.c_float(1e-8), None, fake, None, fake, ctypes.c_size_t(512), None)
    assert rc == lib.OPD_ERR_INVALID_ARG
    rc = lib.call_raw("opd_seq_mean_token_mean_device", fake, fake, ctypes.c_int64(4), ctypes.c_int64(2),
                      ctypes.c_float(-1.0), None, fake, None, fake, ctypes.c_size_t(4096), None)
    assert rc == lib.OPD_ERR_INVALID_ARG


def test_seq_mean_counts_arguments(lib):
    vp = ctypes.c_void_p
    fake = vp(1 << 20)
    n = ctypes.c_size_t(lib.opd_seq_mean_token_mean_workspace_size(8))
    counts = lambda T, n_ids, c: lib.call_raw("opd_seq_mean_token_mean_counts", fake, fake, ctypes.c_int64(T),
                                              ctypes.c_int64(n_ids), c, fake, n, None)
    assert counts(4, 0, fake) == lib.OPD_ERR_INVALID_ARG
    assert counts(4, 8, None) == lib.OPD_ERR_INVALID_ARG
    assert counts(-1, 8, fake) == lib.OPD_ERR_INVALID_ARG
    assert lib.call_raw("opd_seq_mean_token_mean_counts", fake, fake, ctypes.c_int64(4), ctypes.c_int64(8), fake,
                        fake, ctypes.c_size_t(64), None) == lib.OPD_ERR_INVALID_ARG  # workspace too small

    def from_counts(T, loss_in, w_out, loss_out, eps=1e-8):
        return lib.call_raw("opd_seq_mean_token_mean_from_counts", fake, fake, ctypes.c_int64(T), ctypes.c_int64(8),
                            fake, ctypes.c_float(eps), loss_in, w_out, loss_out, fake, n, None)
    assert from_counts(4, None, None, None) == lib.OPD_ERR_INVALID_ARG  # nothing requested
    assert from_counts(4, None, None, fake) == lib.OPD_ERR_INVALID_ARG  # a loss of rows without their losses
    assert from_counts(4, fake, fake, None, eps=-1.0) == lib.OPD_ERR_INVALID_ARG
    # no rows: the loss needs no input (the call then stops at the missing GPU, or runs)
    assert from_counts(0, None, None, fake) != lib.OPD_ERR_INVALID_ARG


def test_kl_seq_mean_arguments(lib):
    p = lib.make_problem(1000, 64, 64, 500, lib.OPD_DTYPE_BF16, 1.0)
    base = lib.opd_kl_workspace_size(p)
    assert lib.opd_kl_seq_mean_workspace_size(p, 10) >= base + 4 * 1000 + 16 + 80
    assert lib.opd_kl_seq_mean_workspace_size(p, 0) == 0
    assert lib.opd_kl_seq_mean_workspace_size(lib.make_problem(8, 12, 8, 8), 4) == 0
    vp = ctypes.c_void_p
    fake = vp(1 << 20)
    n = ctypes.c_size_t(lib.opd_kl_seq_mean_workspace_size(p, 10))
    args = lambda n_ids, eps, loss: [ctypes.byref(p), fake, fake, fake, fake, fake, fake, ctypes.c_int64(n_ids),
                                     ctypes.c_float(eps), loss, fake, fake, fake, fake, 0, fake, n, None]
    assert lib.call_raw("opd_kl_seq_mean_fwd_bwd", *args(0, 1e-8, fake)) == lib.OPD_ERR_INVALID_ARG
    assert lib.call_raw("opd_kl_seq_mean_fwd_bwd", *args(10, -1.0, fake)) == lib.OPD_ERR_INVALID_ARG
    assert lib.call_raw("opd_kl_seq_mean_fwd_bwd", *args(10, 1e-8, None)) == lib.OPD_ERR_INVALID_ARG
    small = [ctypes.byref(p), fake, fake, fake, fake, fake, fake, ctypes.c_int64(10), ctypes.c_float(1e-8), fake,
             fake, fake, fake, fake, 0, fake, ctypes.c_size_t(base), None]
    assert lib.call_raw("opd_kl_seq_mean_fwd_bwd", *small) == lib.OPD_ERR_INVALID_ARG  # KL workspace only


def test_binding_checks_every_buffer_before_the_call(lib):
    """The C entry points see bare pointers, so the Python binding checks each buffer's
    element type, contiguity and size against the problem before calling. The checks run
    before the CUDA-device check, so host tensors exercise them here."""
    import torch
    T, d_s, d_t, V = 8, 16, 24, 40
    prob = lib.make_problem(T, d_s, d_t, V, lib.OPD_DTYPE_BF16, 1.0)
    bf = lambda *s: torch.zeros(*s, dtype=torch.bfloat16)
    f32 = lambda *s: torch.zeros(*s, dtype=torch.float32)
    mask = torch.ones(T, dtype=torch.uint8)
    ws = torch.zeros(64, dtype=torch.uint8)
    good = dict(H_s=bf(T, d_s), H_t=bf(T, d_t), W_s=bf(V, d_s), W_t=bf(V, d_t), mask=mask, kl_out=f32(T),
                stats=f32(T, 3), workspace=ws)

    def call(**over):
        a = dict(good, **over)
        lib.opd_kl_forward(prob, a["H_s"], a["H_t"], a["W_s"], a["W_t"], a["mask"], a["kl_out"], a["stats"],
                           a["workspace"])

    with pytest.raises(TypeError, match="H_s: dtype torch.float32"):
        call(H_s=f32(T, d_s))
    with pytest.raises(ValueError, match="W_t holds"):
        call(W_t=bf(V - 1, d_t))
    with pytest.raises(ValueError, match="stats holds"):
        call(stats=f32(T, 2))
    with pytest.raises(ValueError, match="H_t: buffers must be contiguous"):
        call(H_t=bf(d_t, T).t())
    with pytest.raises(TypeError, match="mask: dtype torch.int64"):
        call(mask=torch.ones(T, dtype=torch.int64))
    with pytest.raises(ValueError, match="must be CUDA tensors"):
        call()  # every size and type right: only the device is wrong
    with pytest.raises(ValueError, match="must be CUDA tensors"):
        call(mask=torch.ones(T, dtype=torch.bool))  # one byte per row, accepted
    g = f32(T)
    with pytest.raises(ValueError, match="dW_s holds"):
        lib.opd_kl_fwd_bwd(prob, good["H_s"], good["H_t"], good["W_s"], good["W_t"], mask, g, f32(T), f32(T, 3),
                           f32(T, d_s), f32(V, d_s - 1), False, ws)
    with pytest.raises(TypeError, match="tokens: dtype torch.int64"):
        lib.opd_score_tokens(prob, good["H_s"], good["W_s"], torch.zeros(T, dtype=torch.int64), mask, f32(T),
                             f32(T), ws)
    with pytest.raises(TypeError, match="seg_id: dtype torch.int64"):
        lib.opd_seq_mean_token_mean_device(torch.zeros(T, dtype=torch.int64), mask, 1, 1e-8, None, f32(T), None, ws)
    f32p = lib.make_problem(T, d_s, d_t, V, lib.OPD_DTYPE_F32, 1.0)
    with pytest.raises(TypeError, match="H_s: dtype torch.bfloat16"):
        lib.opd_kl_forward(f32p, good["H_s"], f32(T, d_t), f32(V, d_s), f32(V, d_t), mask, f32(T), f32(T, 3), ws)


def test_row_chunk_sizing_for_a_workspace_budget(lib):
    from paper_2609_36608_gb300 import chunking
    p = lib.make_problem(16384, 2048, 4096, 151936, lib.OPD_DTYPE_BF16, 1.0)
    full = lib.opd_kl_workspace_size(p)
    assert chunking.max_rows_for_workspace(p, full) == 16384
    for budget in (1 << 30, 2 << 30, full - 1):
        rows = chunking.max_rows_for_workspace(p, budget)
        assert rows % 256 == 0 and 0 < rows < 16384
        fits = lambda r: lib.opd_kl_workspace_size(lib.make_problem(r, 2048, 4096, 151936, 0, 1.0)) <= budget
        assert fits(rows) and not fits(rows + 256)
    assert chunking.max_rows_for_workspace(p, 1 << 20) == 0
    small = lib.make_problem(100, 64, 64, 500, lib.OPD_DTYPE_BF16, 1.0)
    assert chunking.max_rows_for_workspace(small, lib.opd_kl_workspace_size(small)) == 100
