"""torch.autograd entry points over the C ABI (argument marshalling only; every step runs
in libopdkl.so).

OPDReverseKL: per-token reverse KL(student || teacher) of Section 3, Eq. reverse-kl, masked
to supervised rows; its backward calls opd_kl_backward with the upstream per-token gradient.
The teacher is frozen (Appendix B.4), so H_t and W_t get no gradient.

OPDSeqMeanKLLoss: the paper's batch loss over the per-token KL (Appendix B.4,
seq-mean-token-mean), computed with its gradients by one opd_kl_seq_mean_fwd_bwd call in
the forward; the backward scales those gradients by the upstream scalar.

OPDSurrogateLoss: the sampled-token dual-clip surrogate the paper optimises (Appendix B.4,
Eq. opd-token-advantage, opd-ratio, opd-dual-clip, opd-surrogate) with seq-mean-token-mean
weights computed on the device; one opd_surrogate_fwd_bwd call in the forward, the
backward scales its gradients. score_tokens: the frozen teacher's log-partition and token
log-probabilities (no gradient).

Gradients come back in the dtype of the tensors they belong to (autograd's rule); the
library computes them in float32.

Errors found on the device (a token id outside [0, V), a response id >= n_ids, a bounded
wait that ran out) set a status word in the call's workspace; these functions do not read
it, so outside debug mode such a call returns a wrong loss without raising. With
OPD_KL_SYNC_CHECK=1 in the environment every library call synchronises, reads that word
and scans its outputs for NaN and infinity, and the binding raises OpdError.
"""

from __future__ import annotations

import torch

from . import opd_kl


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return opd_kl.OPD_DTYPE_BF16
    if t.dtype == torch.float32:
        return opd_kl.OPD_DTYPE_F32
    raise TypeError(f"hidden states and heads must be bfloat16 or float32, not {t.dtype}")


def _problem(H_s, H_t, W_s, W_t, temperature):
    if not (H_s.dtype == H_t.dtype == W_s.dtype == W_t.dtype):
        raise TypeError("H_s, H_t, W_s and W_t must share one dtype")
    return opd_kl.make_problem(H_s.shape[0], H_s.shape[1], H_t.shape[1], W_s.shape[0], _dtype_code(H_s),
                               float(temperature))


def _contig(*ts):
    return [t.contiguous() for t in ts]


class OPDReverseKL(torch.autograd.Function):
    """kl = OPDReverseKL.apply(H_s, H_t, W_s, W_t, mask, temperature) -> [T] float32."""

    @staticmethod
    def forward(ctx, H_s, H_t, W_s, W_t, mask, temperature=1.0):
        H_s, H_t, W_s, W_t = _contig(H_s, H_t, W_s, W_t)
        mask = mask.to(torch.uint8).contiguous()
        prob = _problem(H_s, H_t, W_s, W_t, temperature)
        # the forward needs only the leading part of the workspace (no dz buffer); the
        # backward takes a full one, so the T x V dz memory is held only while it runs
        ws = opd_kl.allocate_workspace(prob, H_s.device, forward_only=True)
        T = H_s.shape[0]
        kl = torch.empty(T, device=H_s.device, dtype=torch.float32)
        stats = torch.empty(T, 3, device=H_s.device, dtype=torch.float32)
        opd_kl.opd_kl_forward(prob, H_s, H_t, W_s, W_t, mask, kl, stats, ws)
        ctx.save_for_backward(H_s, H_t, W_s, W_t, mask, stats)
        ctx.temperature = float(temperature)
        return kl

    @staticmethod
    def backward(ctx, grad_kl):
        H_s, H_t, W_s, W_t, mask, stats = ctx.saved_tensors
        prob = _problem(H_s, H_t, W_s, W_t, ctx.temperature)
        ws = opd_kl.allocate_workspace(prob, H_s.device)
        dH = torch.empty(H_s.shape, device=H_s.device, dtype=torch.float32)
        dW = torch.empty(W_s.shape, device=W_s.device, dtype=torch.float32)
        opd_kl.opd_kl_backward(prob, H_s, H_t, W_s, W_t, mask, stats, grad_kl.float().contiguous(), dH, dW, False, ws)
        return dH.to(H_s.dtype), None, dW.to(W_s.dtype), None, None, None


class OPDSeqMeanKLLoss(torch.autograd.Function):
    """loss = OPDSeqMeanKLLoss.apply(H_s, H_t, W_s, W_t, mask, seg_id, n_ids, temperature, eps)
    -> scalar float32: L = sum_i w_i KL_i with the paper's seq-mean-token-mean weights."""

    @staticmethod
    def forward(ctx, H_s, H_t, W_s, W_t, mask, seg_id, n_ids, temperature=1.0, eps=1e-8):
        H_s, H_t, W_s, W_t = _contig(H_s, H_t, W_s, W_t)
        mask = mask.to(torch.uint8).contiguous()
        seg_id = seg_id.to(torch.int32).contiguous()
        prob = _problem(H_s, H_t, W_s, W_t, temperature)
        ws = opd_kl.allocate_seq_mean_workspace(prob, int(n_ids), H_s.device)
        T = H_s.shape[0]
        dev = H_s.device
        loss = torch.empty(1, device=dev, dtype=torch.float32)
        kl = torch.empty(T, device=dev, dtype=torch.float32)
        stats = torch.empty(T, 3, device=dev, dtype=torch.float32)
        dH = torch.empty(H_s.shape, device=dev, dtype=torch.float32)
        dW = torch.empty(W_s.shape, device=dev, dtype=torch.float32)
        opd_kl.opd_kl_seq_mean_fwd_bwd(prob, H_s, H_t, W_s, W_t, mask, seg_id, int(n_ids), float(eps), loss, kl,
                                       stats, dH, dW, False, ws)
        ctx.save_for_backward(dH, dW)
        ctx.dtypes = (H_s.dtype, W_s.dtype)
        return loss[0]

    @staticmethod
    def backward(ctx, grad_loss):
        dH, dW = ctx.saved_tensors
        g = grad_loss.float()
        return (dH * g).to(ctx.dtypes[0]), None, (dW * g).to(ctx.dtypes[1]), None, None, None, None, None, None


class OPDSurrogateLoss(torch.autograd.Function):
    """loss = OPDSurrogateLoss.apply(H_s, W_s, tokens, logp_old, logp_teacher, mask, seg_id, n_ids,
    temperature, eps) -> scalar float32: L = sum_i w_i l_i, with l_i the dual-clip surrogate of token i
    and w the seq-mean-token-mean weights (paper's constants delta = 0.2, kappa = 3, clip 20)."""

    @staticmethod
    def forward(ctx, H_s, W_s, tokens, logp_old, logp_teacher, mask, seg_id, n_ids, temperature=1.0, eps=1e-8):
        if H_s.dtype != torch.bfloat16 or W_s.dtype != torch.bfloat16:
            raise TypeError("the surrogate path takes bfloat16 H_s and W_s")
        H_s, W_s = _contig(H_s, W_s)
        dev = H_s.device
        T, d = H_s.shape
        mask = mask.to(torch.uint8).contiguous()
        seg_id = seg_id.to(torch.int32).contiguous()
        tokens = tokens.to(torch.int32).contiguous()
        logp_old = logp_old.float().contiguous()
        logp_teacher = logp_teacher.float().contiguous()
        prob = opd_kl.make_problem(T, d, d, W_s.shape[0], opd_kl.OPD_DTYPE_BF16, float(temperature))
        ws = opd_kl.allocate_workspace(prob, dev)
        seq_ws = torch.empty(opd_kl.opd_seq_mean_token_mean_workspace_size(int(n_ids)), dtype=torch.uint8,
                             device=dev)
        weights = torch.empty(T, device=dev, dtype=torch.float32)
        loss_tok = torch.empty(T, device=dev, dtype=torch.float32)
        logp = torch.empty(T, device=dev, dtype=torch.float32)
        dH = torch.empty(H_s.shape, device=dev, dtype=torch.float32)
        dW = torch.empty(W_s.shape, device=dev, dtype=torch.float32)
        total = torch.empty(1, device=dev, dtype=torch.float32)
        opd_kl.opd_seq_mean_token_mean_device(seg_id, mask, int(n_ids), float(eps), None, weights, None, seq_ws)
        opd_kl.opd_surrogate_fwd_bwd(prob, H_s, W_s, tokens, logp_old, logp_teacher, mask, weights, loss_tok, logp,
                                     dH, dW, False, ws)
        opd_kl.opd_seq_mean_token_mean_device(seg_id, mask, int(n_ids), float(eps), loss_tok, None, total, seq_ws)
        ctx.save_for_backward(dH, dW)
        ctx.dtypes = (H_s.dtype, W_s.dtype)
        return total[0]

    @staticmethod
    def backward(ctx, grad_loss):
        dH, dW = ctx.saved_tensors
        g = grad_loss.float()
        return (dH * g).to(ctx.dtypes[0]), (dW * g).to(ctx.dtypes[1]), None, None, None, None, None, None, None, None


@torch.no_grad()
def score_tokens(H, W, tokens, mask, temperature=1.0):
    """(lse, logp) of the given tokens under one head (the frozen teacher's scores): float32 [T] each,
    zeros on rows with mask 0."""
    if H.dtype != torch.bfloat16 or W.dtype != torch.bfloat16:
        raise TypeError("scoring takes bfloat16 H and W")
    H, W = _contig(H, W)
    T, d = H.shape
    prob = opd_kl.make_problem(T, d, d, W.shape[0], opd_kl.OPD_DTYPE_BF16, float(temperature))
    ws = opd_kl.allocate_workspace(prob, H.device, forward_only=True)
    lse = torch.empty(T, device=H.device, dtype=torch.float32)
    logp = torch.empty(T, device=H.device, dtype=torch.float32)
    opd_kl.opd_score_tokens(prob, H, W, tokens.to(torch.int32).contiguous(), mask.to(torch.uint8).contiguous(), lse,
                            logp, ws)
    return lse, logp
