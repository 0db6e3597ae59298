"""One on-policy ACRL pass over a batch: the five C-ABI calls in order on one
stream, with every buffer allocated once per batch shape.

    token_stats -> seq_discrepancy -> grpo_advantage -> controller_step
                -> loss_grad_logits

The weights need Y_g, which needs every row of the prompt, so the gradient
pass can only start after the statistics pass has seen the whole batch: the
logits are streamed twice (2 + 4 bytes per element).  For batches whose
gradient does not fit beside the logits, `run(..., chunk_rows=k)` runs the
gradient pass k rows at a time into a chunk-sized buffer and hands each chunk
to a callback.
"""

from __future__ import annotations

import ctypes
from dataclasses import dataclass
from typing import Callable

import torch

from . import api
from ._abi import BATCH_DTYPE, GRP_DTYPE, SEQ_DTYPE, STATE_DTYPE, AcrlError, Params


class AcrlStep:
    def __init__(self, T: int, V: int, ld: int, S: int, Gn: int, params: Params, device="cuda",
                 grad_rows: int | None = None):
        dev = torch.device(device)
        f32 = dict(dtype=torch.float32, device=dev)
        self.T, self.V, self.ld, self.S, self.Gn = T, V, ld, S, Gn
        self.params = params
        self.lse = torch.empty(T, **f32)
        self.logp = torch.empty(T, **f32)
        self.entropy = torch.empty(T, **f32)
        self.disc = api.Discrepancy(torch.empty(T, **f32), torch.empty(T, **f32),
                                    api.struct_buffer(SEQ_DTYPE, S, dev), api.struct_buffer(GRP_DTYPE, Gn, dev),
                                    api.struct_buffer(BATCH_DTYPE, 1, dev), S, Gn)
        self.adv = torch.empty(S, **f32)
        self.weight = torch.empty(T, **f32)
        self.coef = torch.empty(T, **f32)
        self.alpha = torch.empty(S, **f32)
        self.ent_coef = torch.empty(T, **f32) if params.entropy_coeff > 0 else None
        self.grad = torch.empty((grad_rows if grad_rows else T, ld), dtype=torch.bfloat16, device=dev)
        self.token_loss = torch.empty(T, **f32)
        self.loss = torch.empty(1, **f32)
        self.chunk_loss = torch.empty(1, **f32)
        self.flags = api.new_flags(dev)
        self.state = api.controller_init(params, device=dev)

    def reset_controller(self, stream=None):
        api.controller_init(self.params, state=self.state, stream=stream)

    def statistics(self, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, stream=None,
                   exchange: Callable[[torch.Tensor], None] | None = None):
        """Everything up to and including the controller (one read of the logits).
        `exchange`, if given, is applied to the batch-statistics bytes before the
        controller (e.g. distributed.allreduce_batch_stats across ranks)."""
        p = self.params
        api.token_stats(logits, ids, mask, V=self.V, lse=self.lse, logp=self.logp, entropy=self.entropy,
                        flags=self.flags, stream=stream)
        api.seq_discrepancy(self.logp, logp_mu, mask, seq_offsets, group_offsets, self.entropy, out=self.disc,
                            flags=self.flags, stream=stream)
        if exchange is not None:
            exchange(self.disc.batch)
        api.grpo_advantage(rewards, group_offsets, p, adv=self.adv, flags=self.flags, stream=stream)
        api.controller_step(self.state, p, self.disc, mask, seq_offsets, group_offsets, self.adv,
                            weight=self.weight, coef=self.coef, alpha=self.alpha, ent_coef=self.ent_coef,
                            flags=self.flags, stream=stream)

    def gradient(self, logits, ids, mask, stream=None, old_logp=None, recompute_lse=False,
                 chunk_rows: int | None = None, on_chunk: Callable[[int, int, torch.Tensor], None] | None = None):
        """The loss and dL/dlogits (second read of the logits, one write)."""
        lse = None if recompute_lse else self.lse
        eps = self.params.clip_eps
        ent = self.ent_coef is not None
        if not chunk_rows:
            api.loss_grad_logits(logits, ids, mask, lse, old_logp, self.coef, eps, V=self.V,
                                 entropy=self.entropy if ent else None, ent_coef=self.ent_coef, grad=self.grad,
                                 token_loss=self.token_loss, loss=self.loss, flags=self.flags, stream=stream)
            return
        for r0 in range(0, self.T, chunk_rows):
            r1 = min(self.T, r0 + chunk_rows)
            g = self.grad[: r1 - r0]
            api.loss_grad_logits(logits[r0:r1], ids[r0:r1], None if mask is None else mask[r0:r1],
                                 None if lse is None else lse[r0:r1],
                                 None if old_logp is None else old_logp[r0:r1], self.coef[r0:r1], eps, V=self.V,
                                 entropy=self.entropy[r0:r1] if ent else None,
                                 ent_coef=self.ent_coef[r0:r1] if ent else None,
                                 grad=g, token_loss=self.token_loss[r0:r1], loss=self.chunk_loss, flags=self.flags,
                                 stream=stream)
            if on_chunk is not None:
                on_chunk(r0, r1, g)
        api.reduce_loss(self.token_loss, loss=self.loss, stream=stream)

    def run(self, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, stream=None, exchange=None,
            **grad_kw):
        self.statistics(logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, stream=stream,
                        exchange=exchange)
        self.gradient(logits, ids, mask, stream=stream, **grad_kw)

    @classmethod
    def for_batch(cls, batch, params: Params, device="cuda", grad_rows=None):
        return cls(batch.T, batch.V, batch.ld, batch.S, batch.Gn, params, device=device, grad_rows=grad_rows)

    def run_batch(self, batch, stream=None, exchange=None, **grad_kw):
        self.run(batch.logits, batch.ids, batch.mask, batch.logp_mu, batch.rewards, batch.seq_offsets,
                 batch.group_offsets, stream=stream, exchange=exchange, **grad_kw)

    def capture(self, batch, exchange=None, **grad_kw):
        """Record one whole step over `batch`'s buffers as a CUDA graph (the
        kernels' launches only; no host work is left in the step).  Returns the
        torch.cuda.CUDAGraph; `graph.replay()` runs the step again on whatever
        the buffers then hold.  `exchange` must be capturable (e.g. NCCL).
        Capturing runs the step once eagerly first, so it advances the
        controller like any step (it calibrates X on `batch` if X is not yet
        fixed): capture on the first real batch, or call reset_controller()
        afterwards."""
        side = torch.cuda.Stream(device=self.lse.device)
        side.wait_stream(torch.cuda.current_stream(self.lse.device))
        with torch.cuda.stream(side):           # one eager run on the capture stream first
            self.run_batch(batch, exchange=exchange, **grad_kw)
        torch.cuda.current_stream(self.lse.device).wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            self.run_batch(batch, exchange=exchange, **grad_kw)
        return graph

    # host views -----------------------------------------------------------
    def seq_host(self):
        return self.disc.seq_host()

    def grp_host(self):
        return self.disc.grp_host()

    def batch_host(self):
        return self.disc.batch_host()

    def state_host(self):
        return api.read_state(self.state)


@dataclass
class Weights:
    weight: torch.Tensor      # float32 [T] importance weight per token (0 where masked)
    coef: torch.Tensor        # float32 [T] loss coefficient m w A / norm per token
    adv: torch.Tensor         # float32 [S] GRPO advantage per response
    alpha: torch.Tensor       # float32 [S] controller exponent per response
    disc: api.Discrepancy     # lr, d and the per-response / per-prompt / batch statistics
    flags: torch.Tensor       # int32 [1] device flags word of the three calls


def importance_weights(state, params: Params, logp_old, logp_mu, mask, rewards, seq_offsets, group_offsets, *,
                       exchange: Callable[[torch.Tensor], None] | None = None, flags=None, stream=None) -> Weights:
    """The weights of one batch from per-token log-probs alone: the old
    policy's log-probs of the sampled tokens and the rollout engine's (the
    call whose cost Sec. 5.4 reports), i.e. seq_discrepancy, grpo_advantage
    and controller_step in order on one stream.  `state` is the controller
    state (api.controller_init), advanced in place; `exchange` is applied to
    the batch-statistics bytes before the controller, as in
    AcrlStep.statistics."""
    flags = api.new_flags(logp_old.device) if flags is None else flags
    disc = api.seq_discrepancy(logp_old, logp_mu, mask, seq_offsets, group_offsets, flags=flags, stream=stream)
    if exchange is not None:
        exchange(disc.batch)
    adv = api.grpo_advantage(rewards, group_offsets, params, flags=flags, stream=stream)
    weight, coef, alpha = api.controller_step(state, params, disc, mask, seq_offsets, group_offsets, adv, flags=flags,
                                              stream=stream)
    return Weights(weight, coef, adv, alpha, disc, flags)


def _host(t, dtype, n, name):
    if not isinstance(t, torch.Tensor) or t.device.type != "cpu":
        raise AcrlError(f"{name}: expected a host (CPU) tensor")
    if t.dtype != dtype or not t.is_contiguous() or t.numel() < n:
        raise AcrlError(f"{name}: expected a contiguous {dtype} tensor of at least {n} elements")
    return t.data_ptr()


class HostPipeline:
    """acrl_host_pipeline_*: the whole on-policy pass for batches whose inputs
    and outputs are host tensors (page-locked for the copies to overlap),
    with the batch shape (T, V, ld, S, Gn) fixed at construction.  Uploads,
    the five calls and the downloads run chunk by chunk on the library's own
    streams; consecutive steps overlap.  `step` only enqueues: the host
    gradient and loss are valid once `stream` (default: the current stream)
    has been synchronised."""

    def __init__(self, T: int, V: int, ld: int, S: int, Gn: int, chunks: int = 16, device="cuda"):
        nbytes = api.host_pipeline_workspace_bytes(T, ld, S, Gn, chunks)
        if nbytes < 0:
            raise AcrlError("acrl_host_pipeline_workspace_bytes: invalid shape")
        dev = torch.device(device)
        self.device = torch.device("cuda", torch.cuda.current_device()) if dev.index is None else dev
        self.T, self.V, self.ld, self.S, self.Gn, self.chunks = T, V, ld, S, Gn, chunks
        self.handle = ctypes.c_void_p()
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.device)
        self.handle = api.host_pipeline_create(T, V, ld, S, Gn, chunks, self.workspace)

    def batch_stats(self) -> torch.Tensor:
        """The device bytes of the pipeline's acrl_batch_stats (a view into the workspace)."""
        off = api.host_pipeline_batch_stats(self.handle) - self.workspace.data_ptr()
        return self.workspace[off: off + BATCH_DTYPE.itemsize]

    def step(self, state: torch.Tensor, params: Params, logits, ids, mask, logp_mu, rewards, seq_offsets,
             group_offsets, grad, loss, flags: torch.Tensor, stream=None,
             exchange: Callable[[torch.Tensor], None] | None = None) -> None:
        """One step; with `exchange` (e.g. distributed.allreduce_batch_stats) the
        batch-statistics bytes are combined across ranks between the
        discrepancy call and the controller (acrl_host_pipeline_begin, the
        exchange on the stream, acrl_host_pipeline_finish)."""
        if not self.handle:
            raise AcrlError("host pipeline: already closed")
        T, ld, S, Gn = self.T, self.ld, self.S, self.Gn
        if logits.dim() != 2 or logits.shape[0] != T or logits.stride(0) != ld or grad.dim() != 2 or \
                grad.shape[0] != T or grad.stride(0) != ld:
            raise AcrlError(f"logits / grad: expected host bf16 [{T}, {ld}] tensors")
        ptrs = (_host(logits, torch.bfloat16, T * ld, "logits"), _host(ids, torch.int32, T, "ids"),
                None if mask is None else _host(mask, torch.uint8, T, "mask"),
                _host(logp_mu, torch.float32, T, "logp_mu"), _host(rewards, torch.float32, S, "rewards"),
                _host(seq_offsets, torch.int64, S + 1, "seq_offsets"),
                _host(group_offsets, torch.int32, Gn + 1, "group_offsets"),
                _host(grad, torch.bfloat16, T * ld, "grad"), _host(loss, torch.float32, 1, "loss"))
        api._need(state, torch.uint8, STATE_DTYPE.itemsize, "state")
        api._need(flags, torch.int32, 1, "flags")
        if state.device != self.device or flags.device != self.device:
            raise AcrlError("state / flags: expected on the pipeline's device")
        with torch.cuda.device(self.device):
            s = torch.cuda.current_stream(self.device) if stream is None else stream
            if exchange is None:
                api.host_pipeline_step(self.handle, params, state, *ptrs, flags, s)
                return
            api.host_pipeline_begin(self.handle, *ptrs[:7], flags, s)
            with torch.cuda.stream(s):
                exchange(self.batch_stats())
            api.host_pipeline_finish(self.handle, params, state, ptrs[7], ptrs[8], flags, s)

    def close(self) -> None:
        if getattr(self, "handle", None):
            h, self.handle = self.handle, ctypes.c_void_p()
            api.host_pipeline_destroy(h)

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
