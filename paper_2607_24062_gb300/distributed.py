"""Data-parallel use of the ACRL path across ranks (one process per GPU).

Ranks own whole prompts, so every per-token, per-response and per-prompt
quantity is local.  Three numbers are global: the valid-token count N, the
valid-prompt count Q and the sum of Y_g over prompts.  X is the mean of Y_g
over all prompts (Sec. 4.1), and the loss averages over all prompts (or
tokens) of the batch (Eq. grpo_objective), so before acrl_controller_step
each rank sums those three fields of its acrl_batch_stats over the group.
That is the only exchange on the path: three scalars per step.
"""

from __future__ import annotations

import torch
import torch.distributed as dist

from ._abi import BATCH_DTYPE

_OFF = {name: BATCH_DTYPE.fields[name][1] for name in ("n_tokens", "n_groups_valid", "Y_sum")}


def _field(buf: torch.Tensor, name: str, dtype: torch.dtype) -> torch.Tensor:
    off = _OFF[name]
    n = torch.empty((), dtype=dtype).element_size()
    return buf[off:off + n].view(dtype)


def allreduce_batch_stats(batch: torch.Tensor, group=None) -> None:
    """Sum n_tokens, n_groups_valid and Y_sum of one acrl_batch_stats (its
    bytes, on the device the backend uses) over the ranks, in place."""
    if not dist.is_initialized() or dist.get_world_size(group) == 1:
        return
    # one collective: the two counts travel as float64 (exact below 2^53) beside the sum
    fields = (("n_tokens", torch.int64), ("n_groups_valid", torch.int32), ("Y_sum", torch.float64))
    views = [_field(batch, name, dtype) for name, dtype in fields]
    packed = torch.stack([v.reshape(()).to(torch.float64) for v in views])
    dist.all_reduce(packed, op=dist.ReduceOp.SUM, group=group)
    for k, v in enumerate(views):
        v.copy_(packed[k].to(v.dtype))


def shard_seed(base_seed: int, rank: int) -> int:
    """Seed of the batch a rank owns (independent prompts per rank)."""
    return base_seed + 7919 * rank
