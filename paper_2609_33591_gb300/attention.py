"""K-interval attention as a differentiable PyTorch op, and a GPT-2 attention layer on it.

``kint_attention(Q, K, V, cfg)`` is a ``torch.autograd.Function`` over the C ABI: the forward
calls ``kint_attn_fwd`` and keeps the row statistics it writes; the backward calls
``kint_attn_bwd`` with them (Sec. 3 and App. B of the paper: the closed-form backward of
the chosen calibration, reconstruction, surrogate and gradient mode).  Every step runs in
libkint's kernels; PyTorch only allocates and orders the buffers.

``KIntSelfAttention`` is the causal self-attention block of GPT-2 (fused QKV projection,
heads of size C / n_head, output projection) with the softmax replaced by K-interval
attention, the setting the paper trains in.
"""
from __future__ import annotations

import torch

from . import kint


class KIntAttentionFn(torch.autograd.Function):
    """O = KIntAttention(Q, K, V); Q, K, V fp32 CUDA tensors [B, H, T, d], causal."""

    @staticmethod
    def forward(ctx, Q, K, V, cfg: kint.Config, prec: int):
        Q, K, V = (x.contiguous() for x in (Q, K, V))
        O, stats = kint.forward(Q, K, V, cfg, prec)
        ctx.save_for_backward(Q, K, V, O)
        ctx.stats, ctx.cfg, ctx.prec = stats, cfg, prec
        return O

    @staticmethod
    def backward(ctx, dO):
        Q, K, V, O = ctx.saved_tensors
        dQ, dK, dV = kint.backward(Q, K, V, O, dO.contiguous(), ctx.stats, ctx.cfg, ctx.prec)
        return dQ, dK, dV, None, None


def kint_attention(Q, K, V, cfg: kint.Config, prec: int = kint.PREC_TF32):
    """Differentiable causal K-interval attention of fp32 [B, H, T, d] CUDA tensors."""
    return KIntAttentionFn.apply(Q, K, V, cfg, prec)


class KIntSelfAttention(torch.nn.Module):
    """GPT-2 causal self-attention with K-interval attention in place of the softmax:
    x [B, T, C] -> c_attn (C -> 3C) -> n_head heads of C / n_head -> K-interval attention
    -> merge heads -> c_proj (C -> C).  The attention runs in fp32 (the paper trains with fp32
    attention); inputs of another dtype are cast for it and the result cast back."""

    def __init__(self, n_embd: int = 768, n_head: int = 12, cfg: kint.Config | None = None,
                 prec: int = kint.PREC_TF32, bias: bool = True):
        super().__init__()
        if n_embd % n_head:
            raise ValueError("n_embd must be a multiple of n_head")
        self.n_head = n_head
        self.c_attn = torch.nn.Linear(n_embd, 3 * n_embd, bias=bias)
        self.c_proj = torch.nn.Linear(n_embd, n_embd, bias=bias)
        self.cfg = cfg if cfg is not None else kint.Config()
        self.prec = prec

    def forward(self, x):
        B, T, C = x.shape
        H, D = self.n_head, C // self.n_head
        q, k, v = self.c_attn(x).split(C, dim=2)
        q, k, v = (t.view(B, T, H, D).transpose(1, 2).float().contiguous() for t in (q, k, v))
        y = kint_attention(q, k, v, self.cfg, self.prec)
        y = y.to(x.dtype).transpose(1, 2).contiguous().view(B, T, C)
        return self.c_proj(y)
