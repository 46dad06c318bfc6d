"""Differentiable attention on libfbob, twice: ``attention(q, k, v)`` runs the
forward kernel, its backward the first-backward kernels (eqs. 2-3), and the
backward of that backward the BoB kernels (eqs. 4-7).  So
``torch.autograd.grad(..., create_graph=True)`` followed by a second
``torch.autograd.grad`` (a Hessian-vector product through attention) runs
entirely in this library's kernels.

BoB returns the total derivatives of Phi = <dQ,U_Q> + <dK,U_K> + <dV,U_V>
with respect to Q, K, V and dO, the paths through O and L included (Sec. 3.1).
The first-backward node therefore takes O and L as plain, non-differentiable
inputs.  Inputs are contiguous CUDA bf16 tensors [B, H, N, d] with d in
{32, 64, 128, 256}; there is no CPU or PyTorch fallback.
"""
from __future__ import annotations

import math

import torch

from . import attn_bob, attn_bwd, attn_fwd


def _bf16(x: torch.Tensor) -> torch.Tensor:
    return x.to(torch.bfloat16).contiguous()


def _check(q: torch.Tensor) -> None:
    if not q.is_cuda or q.dtype != torch.bfloat16 or q.dim() != 4:
        raise ValueError("fbob attention expects CUDA bf16 tensors of shape [B, H, N, d]")


class _AttnBwd(torch.autograd.Function):
    """(q, k, v, dout) -> (dq, dk, dv); its backward is BoB."""

    @staticmethod
    def forward(ctx, q, k, v, o, lse, dout, scale, causal, window, segments, dropout, blocks):
        dout = _bf16(dout)
        dq, dk, dv, _ = attn_bwd(q, k, v, o, lse, dout, scale, causal, window, segments, dropout,
                                 blocks)
        ctx.save_for_backward(q, k, v, o, lse, dout)
        ctx.scale, ctx.causal, ctx.window, ctx.segments = scale, causal, window, segments
        ctx.dropout, ctx.blocks = dropout, blocks
        return dq, dk, dv

    @staticmethod
    def backward(ctx, gq, gk, gv):
        q, k, v, o, lse, dout = ctx.saved_tensors
        g = [torch.zeros_like(x) if t is None else _bf16(t)
             for t, x in zip((gq, gk, gv), (q, k, v))]
        q_bar, k_bar, v_bar, dout_bar, _ = attn_bob(q, k, v, o, lse, dout, *g, ctx.scale,
                                                    ctx.causal, ctx.window, ctx.segments,
                                                    ctx.dropout, ctx.blocks)
        return q_bar, k_bar, v_bar, None, None, dout_bar, None, None, None, None, None, None


class _Attn(torch.autograd.Function):
    """(q, k, v) -> O = softmax(scale Q K^T + M) V (eq. 1)."""

    @staticmethod
    def forward(ctx, q, k, v, scale, causal, window, segments, dropout, blocks):
        o, lse = attn_fwd(q, k, v, scale, causal, window, segments, dropout, blocks)
        ctx.save_for_backward(q, k, v, o, lse)
        ctx.scale, ctx.causal, ctx.window, ctx.segments = scale, causal, window, segments
        ctx.dropout, ctx.blocks = dropout, blocks
        return o

    @staticmethod
    def backward(ctx, dout):
        q, k, v, o, lse = ctx.saved_tensors
        dq, dk, dv = _AttnBwd.apply(q, k, v, o.detach(), lse, dout, ctx.scale, ctx.causal,
                                    ctx.window, ctx.segments, ctx.dropout, ctx.blocks)
        return dq, dk, dv, None, None, None, None, None, None


def attention(q: torch.Tensor, k: torch.Tensor, v: torch.Tensor, scale: float | None = None,
              causal: bool = False, window: tuple | None = None,
              segments: torch.Tensor | None = None, dropout_p: float = 0.0,
              seed: int = 0, block_mask: torch.Tensor | None = None) -> torch.Tensor:
    """Softmax attention on libfbob, differentiable twice (see the module doc).
    window: (left, right) sliding-window band, -1 = unbounded side; segments:
    int32 CUDA offsets of packed variable-length sequences; dropout_p, seed:
    attention dropout after the softmax with a keep mask regenerated from the
    seed in every kernel (the same mask in the forward and both backwards);
    block_mask: uint8 CUDA [ceil(N/128)]^2 block-sparse mask of 128 x 128
    (query block, key block) tiles, every diagonal block set."""
    for t in (q, k, v):
        _check(t)
    if scale is None:
        scale = 1.0 / math.sqrt(q.shape[-1])
    dropout = (float(dropout_p), int(seed)) if dropout_p else None
    return _Attn.apply(q.contiguous(), k.contiguous(), v.contiguous(), float(scale),
                       bool(causal), None if window is None else tuple(window), segments, dropout,
                       block_mask)
