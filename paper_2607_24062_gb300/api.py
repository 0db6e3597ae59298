"""Python binding of the ACRL C ABI: one function per entry point, same names
without the `acrl_` prefix.  Arguments are torch tensors on the current CUDA
device; this layer only checks dtypes/shapes, passes raw pointers and the
current stream, allocates outputs the caller did not provide, and turns a
non-OK status into an exception.  Every step of the computation runs in the
library's kernels."""

from __future__ import annotations

import ctypes
from dataclasses import dataclass

import numpy as np
import torch

from . import _abi
from ._abi import BATCH_DTYPE, GRP_DTYPE, SEQ_DTYPE, STATE_DTYPE, AcrlError, Params, check, lib  # noqa: F401


def _ptr(t: torch.Tensor | None) -> int | None:
    return None if t is None else t.data_ptr()


def _one_device(tensors) -> torch.device:
    """The GPU every buffer of one call lives on (they must agree)."""
    dev = None
    for t in tensors:
        if t is None:
            continue
        if dev is None:
            dev = t.device
        elif t.device != dev:
            raise AcrlError(f"buffers on {dev} and {t.device}: every buffer of a call must be on one GPU")
    if dev is None or dev.type != "cuda":
        raise AcrlError("expected CUDA tensors")
    return dev


def _call(name: str, tensors, stream, *args) -> None:
    """Call entry point `name` with `args` followed by the stream, on the GPU
    that holds `tensors` (the stream defaults to that GPU's current stream)."""
    dev = _one_device(tensors)
    if stream is not None and stream.device != dev:
        raise AcrlError(f"{name}: stream on {stream.device}, buffers on {dev}")
    fn = getattr(lib(), name)
    if dev.index == torch.cuda.current_device():
        s = torch.cuda.current_stream(dev) if stream is None else stream
        check(fn(*args, s.cuda_stream), name)
        return
    with torch.cuda.device(dev):
        s = torch.cuda.current_stream(dev) if stream is None else stream
        check(fn(*args, s.cuda_stream), name)


def _flags(flags, dev):
    return new_flags(dev) if flags is None else _need(flags, torch.int32, 1, "flags")


def _need(t: torch.Tensor, dtype, n: int | None, name: str):
    if not isinstance(t, torch.Tensor):
        raise AcrlError(f"{name}: expected a torch tensor")
    if t.dtype != dtype:
        raise AcrlError(f"{name}: dtype {t.dtype}, expected {dtype}")
    if not t.is_cuda:
        raise AcrlError(f"{name}: must be a CUDA tensor")
    if not t.is_contiguous():
        raise AcrlError(f"{name}: must be contiguous")
    if n is not None and t.numel() < n:
        raise AcrlError(f"{name}: has {t.numel()} elements, needs {n}")
    return t


def _opt(t, dtype, n, name):
    return None if t is None else _need(t, dtype, n, name)


def _rows(x: torch.Tensor, name: str):
    if x.dtype != torch.bfloat16 or x.dim() != 2:
        raise AcrlError(f"{name}: expected a 2-D bfloat16 tensor")
    if not x.is_cuda or x.stride(1) != 1:
        raise AcrlError(f"{name}: must be a CUDA tensor with unit column stride")
    return x.shape[0], x.stride(0)


def struct_buffer(dtype: np.dtype, n: int, device=None) -> torch.Tensor:
    """Device bytes for n ABI structs."""
    return torch.zeros(max(1, n) * dtype.itemsize, dtype=torch.uint8, device=device or "cuda")


def read_structs(buf: torch.Tensor, dtype: np.dtype, n: int) -> np.ndarray:
    return buf[: n * dtype.itemsize].cpu().numpy().view(dtype)


def new_flags(device=None) -> torch.Tensor:
    return torch.zeros(1, dtype=torch.int32, device=device or "cuda")


def token_stats(logits, ids, mask=None, *, V=None, lse=None, logp=None, entropy=None, flags=None, stream=None):
    """acrl_token_stats.  Returns (lse, logp, entropy) float32 [T]."""
    T, ld = _rows(logits, "logits")
    V = ld if V is None else V
    dev = logits.device
    _need(ids, torch.int32, T, "ids")
    _opt(mask, torch.uint8, T, "mask")
    lse = torch.empty(T, dtype=torch.float32, device=dev) if lse is None else _need(lse, torch.float32, T, "lse")
    logp = torch.empty(T, dtype=torch.float32, device=dev) if logp is None else _need(logp, torch.float32, T, "logp")
    entropy = torch.empty(T, dtype=torch.float32, device=dev) if entropy is None else \
        _need(entropy, torch.float32, T, "entropy")
    flags = _flags(flags, dev)
    _call("acrl_token_stats", (logits, ids, mask, lse, logp, entropy, flags), stream, _ptr(logits), T, V, ld,
          _ptr(ids), _ptr(mask), _ptr(lse), _ptr(logp), _ptr(entropy), _ptr(flags))
    return lse, logp, entropy


@dataclass
class Discrepancy:
    lr: torch.Tensor
    d: torch.Tensor
    seq: torch.Tensor    # device bytes of acrl_seq_stats[S]
    grp: torch.Tensor    # device bytes of acrl_group_stats[Gn]
    batch: torch.Tensor  # device bytes of acrl_batch_stats
    S: int
    Gn: int

    def seq_host(self):
        return read_structs(self.seq, SEQ_DTYPE, self.S)

    def grp_host(self):
        return read_structs(self.grp, GRP_DTYPE, self.Gn)

    def batch_host(self):
        return read_structs(self.batch, BATCH_DTYPE, 1)[0]


def seq_discrepancy(logp_pi, logp_mu, mask, seq_offsets, group_offsets, entropy=None, *, out: Discrepancy | None = None,
                    flags=None, stream=None) -> Discrepancy:
    """acrl_seq_discrepancy."""
    T = logp_pi.numel()
    S = seq_offsets.numel() - 1
    Gn = group_offsets.numel() - 1
    dev = logp_pi.device
    _need(logp_pi, torch.float32, T, "logp_pi")
    _need(logp_mu, torch.float32, T, "logp_mu")
    _opt(mask, torch.uint8, T, "mask")
    _need(seq_offsets, torch.int64, S + 1, "seq_offsets")
    _need(group_offsets, torch.int32, Gn + 1, "group_offsets")
    _opt(entropy, torch.float32, T, "entropy")
    if out is None:
        out = Discrepancy(torch.empty(T, dtype=torch.float32, device=dev), torch.empty(T, dtype=torch.float32, device=dev),
                          struct_buffer(SEQ_DTYPE, S, dev), struct_buffer(GRP_DTYPE, Gn, dev),
                          struct_buffer(BATCH_DTYPE, 1, dev), S, Gn)
    flags = _flags(flags, dev)
    _call("acrl_seq_discrepancy", (logp_pi, logp_mu, mask, seq_offsets, group_offsets, entropy, out.lr, out.d,
                                   out.seq, out.grp, out.batch, flags), stream,
          _ptr(logp_pi), _ptr(logp_mu), _ptr(mask), T, _ptr(seq_offsets), S, _ptr(group_offsets), Gn, _ptr(entropy),
          _ptr(out.lr), _ptr(out.d), _ptr(out.seq), _ptr(out.grp), _ptr(out.batch), _ptr(flags))
    return out


def grpo_advantage(rewards, group_offsets, params: Params, *, adv=None, flags=None, stream=None):
    """acrl_grpo_advantage.  Returns adv float32 [S]."""
    S = rewards.numel()
    Gn = group_offsets.numel() - 1
    _need(rewards, torch.float32, S, "rewards")
    _need(group_offsets, torch.int32, Gn + 1, "group_offsets")
    adv = torch.empty(S, dtype=torch.float32, device=rewards.device) if adv is None else _need(adv, torch.float32, S, "adv")
    flags = _flags(flags, rewards.device)
    _call("acrl_grpo_advantage", (rewards, group_offsets, adv, flags), stream, _ptr(rewards), _ptr(group_offsets), Gn,
          S, ctypes.byref(params), _ptr(adv), _ptr(flags))
    return adv


def controller_init(params: Params, state=None, device=None, stream=None) -> torch.Tensor:
    """acrl_controller_init; allocates the 48-byte device state if not given."""
    state = struct_buffer(STATE_DTYPE, 1, device) if state is None else state
    _need(state, torch.uint8, STATE_DTYPE.itemsize, "state")
    _call("acrl_controller_init", (state,), stream, _ptr(state), ctypes.byref(params))
    return state


def read_state(state: torch.Tensor) -> np.void:
    return read_structs(state, STATE_DTYPE, 1)[0]


def save_state(state: torch.Tensor, stream=None) -> bytes:
    """acrl_controller_save: the controller state's 48 bytes, for a checkpoint
    (the state is plain data)."""
    _need(state, torch.uint8, STATE_DTYPE.itemsize, "state")
    buf = ctypes.create_string_buffer(STATE_DTYPE.itemsize)
    _call("acrl_controller_save", (state,), stream, _ptr(state), ctypes.addressof(buf))
    return buf.raw


def load_state(blob: bytes, state: torch.Tensor | None = None, device=None, stream=None) -> torch.Tensor:
    """acrl_controller_load: restore a state saved by save_state; resuming
    from it is bit-exact."""
    if len(blob) != STATE_DTYPE.itemsize:
        raise AcrlError("controller state: wrong size")
    state = struct_buffer(STATE_DTYPE, 1, device) if state is None else \
        _need(state, torch.uint8, STATE_DTYPE.itemsize, "state")
    buf = ctypes.create_string_buffer(bytes(blob), STATE_DTYPE.itemsize)
    _call("acrl_controller_load", (state,), stream, _ptr(state), ctypes.addressof(buf))
    return state


def controller_step(state, params: Params, disc: Discrepancy, mask, seq_offsets, group_offsets, adv, *, weight=None,
                    coef=None, alpha=None, ent_coef=None, flags=None, stream=None):
    """acrl_controller_step.  Returns (weight [T], coef [T], alpha [S]); the
    entropy-bonus factors go to `ent_coef` [T] when given."""
    T = disc.lr.numel()
    dev = disc.lr.device
    weight = torch.empty(T, dtype=torch.float32, device=dev) if weight is None else _need(weight, torch.float32, T, "weight")
    coef = torch.empty(T, dtype=torch.float32, device=dev) if coef is None else _need(coef, torch.float32, T, "coef")
    alpha = torch.empty(disc.S, dtype=torch.float32, device=dev) if alpha is None else \
        _need(alpha, torch.float32, disc.S, "alpha")
    _need(adv, torch.float32, disc.S, "adv")
    _opt(mask, torch.uint8, T, "mask")
    _opt(ent_coef, torch.float32, T, "ent_coef")
    _need(state, torch.uint8, STATE_DTYPE.itemsize, "state")
    flags = _flags(flags, dev)
    _call("acrl_controller_step", (state, disc.lr, mask, seq_offsets, group_offsets, disc.seq, disc.grp, disc.batch,
                                   adv, weight, coef, alpha, ent_coef, flags), stream,
          _ptr(state), ctypes.byref(params), _ptr(disc.lr), _ptr(mask), T, _ptr(seq_offsets), disc.S,
          _ptr(group_offsets), disc.Gn, _ptr(disc.seq), _ptr(disc.grp), _ptr(disc.batch), _ptr(adv), _ptr(weight),
          _ptr(coef), _ptr(alpha), _ptr(ent_coef), _ptr(flags))
    return weight, coef, alpha


def loss_grad_logits(logits, ids, mask, lse, old_logp, coef, clip_eps: float, *, V=None, entropy=None, ent_coef=None,
                     grad=None, token_loss=None, loss=None, flags=None, stream=None):
    """acrl_loss_grad_logits.  Returns (grad bf16 [T, ld], token_loss [T], loss [1]).
    `entropy` and `ent_coef` (both or neither) add the entropy bonus."""
    T, ld = _rows(logits, "logits")
    V = ld if V is None else V
    dev = logits.device
    _need(ids, torch.int32, T, "ids")
    _opt(mask, torch.uint8, T, "mask")
    _opt(lse, torch.float32, T, "lse")
    _opt(old_logp, torch.float32, T, "old_logp")
    _need(coef, torch.float32, T, "coef")
    _opt(entropy, torch.float32, T, "entropy")
    _opt(ent_coef, torch.float32, T, "ent_coef")
    if grad is None:
        grad = torch.empty((T, ld), dtype=torch.bfloat16, device=dev)
    elif grad.dtype != torch.bfloat16 or grad.dim() != 2 or grad.stride(0) != ld or grad.stride(1) != 1 or \
            grad.shape[0] < T:
        raise AcrlError("grad: expected a bf16 [T, ld] tensor with the logits' row stride")
    token_loss = torch.empty(T, dtype=torch.float32, device=dev) if token_loss is None else \
        _need(token_loss, torch.float32, T, "token_loss")
    loss = torch.empty(1, dtype=torch.float32, device=dev) if loss is None else _need(loss, torch.float32, 1, "loss")
    flags = _flags(flags, dev)
    _call("acrl_loss_grad_logits", (logits, ids, mask, lse, old_logp, coef, entropy, ent_coef, grad, token_loss, loss,
                                    flags), stream,
          _ptr(logits), T, V, ld, _ptr(ids), _ptr(mask), _ptr(lse), _ptr(old_logp), _ptr(coef), _ptr(entropy),
          _ptr(ent_coef), float(clip_eps), _ptr(grad), _ptr(token_loss), _ptr(loss), _ptr(flags))
    return grad, token_loss, loss


def reduce_loss(token_loss, *, loss=None, stream=None):
    """acrl_reduce_loss."""
    T = token_loss.numel()
    _need(token_loss, torch.float32, T, "token_loss")
    loss = torch.empty(1, dtype=torch.float32, device=token_loss.device) if loss is None else \
        _need(loss, torch.float32, 1, "loss")
    _call("acrl_reduce_loss", (token_loss, loss), stream, _ptr(token_loss), T, _ptr(loss))
    return loss


def lmhead_workspace_bytes(M: int, N: int) -> int:
    return int(lib().acrl_lmhead_workspace_bytes(M, N))


def lmhead_logits_stats(hidden, weight, *, N=None, logits=None, partials=None, flags=None, stream=None):
    """acrl_lmhead_logits_stats.  hidden bf16 [M, K], weight bf16 [N, K].
    Returns (logits bf16 [M, ldl], partials workspace)."""
    M, ldh = _rows(hidden, "hidden")
    Nw, ldw = _rows(weight, "weight")
    N = Nw if N is None else N
    K = hidden.shape[1]
    if weight.shape[1] != K:
        raise AcrlError("hidden and weight disagree on K")
    dev = hidden.device
    ldl = ((N + 7) // 8) * 8
    if logits is None:
        logits = torch.empty((M, ldl), dtype=torch.bfloat16, device=dev)
    else:
        _, ldl = _rows(logits, "logits")
    nbytes = lmhead_workspace_bytes(M, N)
    if partials is None:
        partials = torch.empty(max(1, nbytes // 4), dtype=torch.float32, device=dev)
    else:
        _need(partials, torch.float32, (nbytes + 3) // 4, "partials")
    flags = _flags(flags, dev)
    _call("acrl_lmhead_logits_stats", (hidden, weight, logits, partials, flags), stream, _ptr(hidden), M, K, ldh,
          _ptr(weight), N, ldw, _ptr(logits), ldl, _ptr(partials), _ptr(flags))
    return logits, partials


def lmhead_merge(partials, logits, ids, mask=None, *, N=None, lse=None, logp=None, entropy=None, flags=None,
                 stream=None):
    """acrl_lmhead_merge.  Returns (lse, logp, entropy)."""
    M, ldl = _rows(logits, "logits")
    N = ldl if N is None else N
    dev = logits.device
    _need(ids, torch.int32, M, "ids")
    _opt(mask, torch.uint8, M, "mask")
    lse = torch.empty(M, dtype=torch.float32, device=dev) if lse is None else _need(lse, torch.float32, M, "lse")
    logp = torch.empty(M, dtype=torch.float32, device=dev) if logp is None else _need(logp, torch.float32, M, "logp")
    entropy = torch.empty(M, dtype=torch.float32, device=dev) if entropy is None else \
        _need(entropy, torch.float32, M, "entropy")
    _need(partials, torch.float32, (lmhead_workspace_bytes(M, N) + 3) // 4, "partials")
    flags = _flags(flags, dev)
    _call("acrl_lmhead_merge", (partials, logits, ids, mask, lse, logp, entropy, flags), stream, _ptr(partials),
          _ptr(logits), M, N, ldl, _ptr(ids), _ptr(mask), _ptr(lse), _ptr(logp), _ptr(entropy), _ptr(flags))
    return lse, logp, entropy


def lmhead_stats_noalloc(hidden, weight, ids, mask=None, *, N=None, logits=None, lse=None, logp=None, entropy=None,
                         flags=None, stream=None):
    """acrl_lmhead_stats_noalloc (GEMM + merge with the library's fixed scratch).
    Returns (logits, lse, logp, entropy)."""
    M, ldh = _rows(hidden, "hidden")
    Nw, ldw = _rows(weight, "weight")
    N = Nw if N is None else N
    K = hidden.shape[1]
    if weight.shape[1] != K:
        raise AcrlError("hidden and weight disagree on K")
    dev = hidden.device
    if logits is None:
        logits = torch.empty((M, ((N + 7) // 8) * 8), dtype=torch.bfloat16, device=dev)
    _, ldl = _rows(logits, "logits")
    _need(ids, torch.int32, M, "ids")
    _opt(mask, torch.uint8, M, "mask")
    f32 = dict(dtype=torch.float32, device=dev)
    lse = torch.empty(M, **f32) if lse is None else _need(lse, torch.float32, M, "lse")
    logp = torch.empty(M, **f32) if logp is None else _need(logp, torch.float32, M, "logp")
    entropy = torch.empty(M, **f32) if entropy is None else _need(entropy, torch.float32, M, "entropy")
    flags = _flags(flags, dev)
    _call("acrl_lmhead_stats_noalloc", (hidden, weight, logits, ids, mask, lse, logp, entropy, flags), stream,
          _ptr(hidden), M, K, ldh, _ptr(weight), N, ldw, _ptr(logits), ldl, _ptr(ids), _ptr(mask), _ptr(lse),
          _ptr(logp), _ptr(entropy), _ptr(flags))
    return logits, lse, logp, entropy


def selftest_wait_timeout(flags, limit_ns: int, stream=None) -> None:
    """acrl_selftest_wait_timeout: a bounded wait on a barrier nothing arrives on."""
    _need(flags, torch.int32, 1, "flags")
    _call("acrl_selftest_wait_timeout", (flags,), stream, _ptr(flags), int(limit_ns))


def controller_save(state: torch.Tensor, stream=None) -> bytes:
    """acrl_controller_save (the same as save_state)."""
    return save_state(state, stream)


def controller_load(blob: bytes, state: torch.Tensor | None = None, device=None, stream=None) -> torch.Tensor:
    """acrl_controller_load (the same as load_state)."""
    return load_state(blob, state, device, stream)


# The host-buffer pipeline at the level of its handle (pipeline.HostPipeline wraps these).
def host_pipeline_workspace_bytes(T: int, ld: int, S: int, Gn: int, chunks: int) -> int:
    """acrl_host_pipeline_workspace_bytes (-1 for an invalid shape)."""
    return int(lib().acrl_host_pipeline_workspace_bytes(T, ld, S, Gn, chunks))


def host_pipeline_create(T: int, V: int, ld: int, S: int, Gn: int, chunks: int, workspace: torch.Tensor):
    """acrl_host_pipeline_create on a device workspace tensor (on its device).  Returns the handle."""
    _need(workspace, torch.uint8, max(0, host_pipeline_workspace_bytes(T, ld, S, Gn, chunks)), "workspace")
    handle = ctypes.c_void_p()
    with torch.cuda.device(_one_device((workspace,))):
        check(lib().acrl_host_pipeline_create(ctypes.byref(handle), T, V, ld, S, Gn, chunks, workspace.data_ptr(),
                                              workspace.numel()), "acrl_host_pipeline_create")
    return handle


def host_pipeline_step(handle, params: Params, state, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets,
                       grad, loss, flags, stream) -> None:
    """acrl_host_pipeline_step; host arrays as raw addresses (int), device ones as tensors."""
    check(lib().acrl_host_pipeline_step(handle, ctypes.byref(params), _ptr(state), logits, ids, mask, logp_mu,
                                        rewards, seq_offsets, group_offsets, grad, loss, _ptr(flags),
                                        stream.cuda_stream), "acrl_host_pipeline_step")


def host_pipeline_begin(handle, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, flags,
                        stream) -> None:
    """acrl_host_pipeline_begin; host arrays as raw addresses (int)."""
    check(lib().acrl_host_pipeline_begin(handle, logits, ids, mask, logp_mu, rewards, seq_offsets, group_offsets,
                                         _ptr(flags), stream.cuda_stream), "acrl_host_pipeline_begin")


def host_pipeline_finish(handle, params: Params, state, grad, loss, flags, stream) -> None:
    """acrl_host_pipeline_finish; the host gradient and loss as raw addresses (int)."""
    check(lib().acrl_host_pipeline_finish(handle, ctypes.byref(params), _ptr(state), grad, loss, _ptr(flags),
                                          stream.cuda_stream), "acrl_host_pipeline_finish")


def host_pipeline_batch_stats(handle) -> int:
    """acrl_host_pipeline_batch_stats: the device address of the pipeline's batch statistics."""
    return int(lib().acrl_host_pipeline_batch_stats(handle) or 0)


def host_pipeline_destroy(handle) -> None:
    """acrl_host_pipeline_destroy."""
    check(lib().acrl_host_pipeline_destroy(handle), "acrl_host_pipeline_destroy")


def abi_version() -> int:
    """acrl_abi_version."""
    return int(lib().acrl_abi_version())


def status_string(status: int) -> str:
    """acrl_status_string."""
    return lib().acrl_status_string(status).decode()


def struct_size(which: int) -> int:
    """acrl_struct_size."""
    return int(lib().acrl_struct_size(which))


def read_flags(flags, stream=None) -> int:
    """acrl_read_flags (synchronises the stream)."""
    host = ctypes.c_int32(0)
    _need(flags, torch.int32, 1, "flags")
    _call("acrl_read_flags", (flags,), stream, _ptr(flags), ctypes.byref(host))
    return int(host.value)


def check_flags(flags, stream=None) -> None:
    """acrl_check_flags: synchronises the stream and raises AcrlError (naming
    the bits) if any device flag is set."""
    _need(flags, torch.int32, 1, "flags")
    dev = _one_device((flags,))
    with torch.cuda.device(dev):
        s = torch.cuda.current_stream(dev) if stream is None else stream
        st = lib().acrl_check_flags(_ptr(flags), s.cuda_stream)
    if st == _abi.ERR_DEVICE_FLAGS:
        raise AcrlError(f"device flags raised: 0x{read_flags(flags, stream):x}")
    check(st, "acrl_check_flags")


__all__ = ["Params", "AcrlError", "token_stats", "seq_discrepancy", "grpo_advantage", "controller_init",
           "controller_step", "loss_grad_logits", "reduce_loss", "read_flags", "check_flags", "read_state", "Discrepancy",
           "lmhead_logits_stats", "lmhead_merge", "lmhead_workspace_bytes", "lmhead_stats_noalloc", "save_state",
           "load_state", "controller_save", "controller_load", "selftest_wait_timeout",
           "host_pipeline_workspace_bytes", "host_pipeline_create", "host_pipeline_step", "host_pipeline_begin",
           "host_pipeline_finish", "host_pipeline_batch_stats", "host_pipeline_destroy", "abi_version",
           "status_string", "struct_size", "struct_buffer", "read_structs", "new_flags", "_abi"]
