"""The on-policy ACRL loss as a torch.autograd function.

    loss = acrl_loss(step, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets)
    loss.backward()      # dL/dlogits flows into whatever produced the logits

The forward runs the whole pass of `AcrlStep` (statistics, discrepancy,
advantages, controller, then the gradient kernel, which writes dL/dlogits in
bf16 while it computes the loss), so the backward needs no second pass over
the logits: it hands back that buffer, scaled by the incoming gradient when
that is not 1.  The gradient is the one of Eq. ACRL on the on-policy step
(theta = theta_old, so r = 1), with the importance weights treated as
constants, as the paper's rho is built from theta_old.

The returned gradient is a view of `step.grad`: it stays valid until the same
step object runs again.
"""

from __future__ import annotations

from typing import Callable

import torch

from .pipeline import AcrlStep


class _AcrlLoss(torch.autograd.Function):
    @staticmethod
    def forward(ctx, logits, step, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, exchange):
        step.run(logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, exchange=exchange)
        ctx.step = step
        ctx.rows, ctx.cols = logits.shape
        return step.loss.reshape(()).clone()

    @staticmethod
    def backward(ctx, grad_out):
        g = ctx.step.grad[: ctx.rows, : ctx.cols]
        if float(grad_out) != 1.0:  # one scalar read; the common loss.backward() passes 1
            g = g * grad_out.to(g.dtype)
        return g, None, None, None, None, None, None, None, None


def acrl_loss(step: AcrlStep, logits: torch.Tensor, ids, mask, logp_mu, rewards, seq_offsets, group_offsets,
              exchange: Callable[[torch.Tensor], None] | None = None) -> torch.Tensor:
    """The step's scalar loss (fp32, 0-d) with dL/dlogits attached for
    autograd.  `logits` is the bf16 [T, V] tensor `step` was built for (row
    stride `step.ld`); the other arguments are those of `AcrlStep.run`."""
    if logits.shape != (step.T, step.V) or logits.stride(0) != step.ld:
        raise ValueError(f"logits: expected shape ({step.T}, {step.V}) with row stride {step.ld}")
    return _AcrlLoss.apply(logits, step, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, exchange)
