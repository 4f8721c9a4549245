"""The reverse-KL step over row chunks, to bound its workspace (argument marshalling only).

The workspace of opd_kl_fwd_bwd holds the bf16 dz buffer of T_pad x V elements: 5.0 GB at
T = 16,384 and V = 151,936, and 40 GB at T = 131,072. Rows are independent for KL_i and
dH_s[i, :] (Section 3, Eq. reverse-kl), and dW_s sums over the rows. So a batch can run as
consecutive row chunks that share one smaller workspace: each chunk gets its own rows'
upstream weights (computed once for the whole batch, e.g. the seq-mean-token-mean weights),
and every chunk after the first adds its dW_s part to what the buffer holds
(accumulate_dW). The results equal one call over the whole batch, up to the order of the dW_s
sums. The chunks run one after another on one stream, so they reuse the workspace safely.
"""

from __future__ import annotations

from . import opd_kl


def max_rows_for_workspace(problem: opd_kl.opd_problem, budget_bytes: int) -> int:
    """The most rows of `problem` (a multiple of 256, or all T rows) whose opd_kl_fwd_bwd workspace
    fits in budget_bytes; 0 if not even 256 rows fit."""

    def size(rows: int) -> int:
        return opd_kl.opd_kl_workspace_size(opd_kl.make_problem(rows, problem.d_s, problem.d_t, problem.V,
                                                                 problem.dtype, problem.temperature))

    T = int(problem.T)
    if T <= 0 or size(T) <= budget_bytes:
        return max(T, 0)
    lo, hi = 0, (T + 255) // 256  # in units of 256 rows: size(256 lo) fits, size(256 hi) does not
    if size(256) > budget_bytes:
        return 0
    lo = 1
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if size(256 * mid) <= budget_bytes:
            lo = mid
        else:
            hi = mid
    return 256 * lo


def kl_fwd_bwd_in_row_chunks(problem, H_s, H_t, W_s, W_t, mask, grad_kl, kl_out, stats, dH_s, dW_s,
                             accumulate_dW: bool, budget_bytes: int, device="cuda", stream=None) -> int:
    """opd_kl_fwd_bwd over consecutive row chunks whose shared workspace fits budget_bytes; the
    outputs are those of one call over all rows. The workspace is allocated once, through
    PyTorch. Returns the number of chunks. Raises ValueError if not even 256 rows fit."""
    import torch

    T = int(problem.T)
    rows = max_rows_for_workspace(problem, budget_bytes)
    if T > 0 and rows == 0:
        raise ValueError(f"a workspace of {budget_bytes} bytes holds fewer than 256 rows of this problem")
    rows = max(rows, 1)
    chunk = opd_kl.make_problem(min(rows, max(T, 0)), problem.d_s, problem.d_t, problem.V, problem.dtype,
                                problem.temperature)
    ws = torch.empty(opd_kl.opd_kl_workspace_size(chunk), dtype=torch.uint8, device=device)
    n = 0
    for a in range(0, max(T, 1), rows):
        b = min(T, a + rows)
        part = opd_kl.make_problem(b - a, problem.d_s, problem.d_t, problem.V, problem.dtype, problem.temperature)
        opd_kl.opd_kl_fwd_bwd(part, H_s[a:b], H_t[a:b], W_s, W_t, mask[a:b], grad_kl[a:b], kl_out[a:b],
                              stats[a:b], dH_s[a:b], dW_s, bool(accumulate_dW) or n > 0, ws, stream)
        n += 1
    return n
