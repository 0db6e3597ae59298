"""Two ranks sharing this one GPU, each running the real kernels on its own
shard of prompts and exchanging the three batch sums through a gloo process
group (an all-reduce in host code between the calls: no kernel of one rank
waits on the other).  Each rank's X, weights and loss coefficients must equal
the oracle's on the two shards concatenated."""

import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import oracle as O
import workloads as W
from parity import assert_close_rel, oracle_params, rows_f64

pytestmark = pytest.mark.gpu

SPEC = W.small_variant(W.GRPO, name="dist_gpu", n_prompts=3, group_size=4, len_lo=10, len_hi=120, V=3000,
                       perturb_frac=0.4, perturb_std=0.3)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _host(b):
    h = {k: getattr(b, k).cpu().numpy() for k in ("ids", "mask", "seq_offsets", "group_offsets")}
    h["mu"] = b.logp_mu.cpu().numpy().astype(np.float64)
    h["R"] = b.rewards.cpu().numpy().astype(np.float64)
    h["z"] = rows_f64(b.logits, np.arange(b.T), b.V)
    return h


def _rank(rank, world, port, results):
    import torch.distributed as dist

    import paper_2607_24062_gb300 as acrl
    from paper_2607_24062_gb300 import distributed as D
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.cuda.set_device(0)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    b = W.generate(SPEC, seed=D.shard_seed(41, rank), device="cuda")
    step = acrl.AcrlStep.for_batch(b, acrl.Params())
    step.run_batch(b, exchange=D.allreduce_batch_stats)
    torch.cuda.synchronize()
    results[rank] = {"X": float(step.state_host()["X"]), "weight": step.weight.cpu().numpy(),
                     "coef": step.coef.cpu().numpy(), "flags": acrl.read_flags(step.flags), **_host(b)}
    dist.destroy_process_group()


def test_two_ranks_on_one_gpu_match_the_oracle_on_the_whole_batch():
    with mp.get_context("spawn").Manager() as mgr:
        results = mgr.dict()
        mp.start_processes(_rank, args=(2, _free_port(), results), nprocs=2, start_method="spawn")
        res = [dict(results[r]) for r in range(2)]
    assert res[0]["flags"] == 0 and res[1]["flags"] == 0
    cat = np.concatenate
    T0, S0 = len(res[0]["ids"]), len(res[0]["seq_offsets"]) - 1
    so = cat([res[0]["seq_offsets"], res[1]["seq_offsets"][1:] + T0])
    go = cat([res[0]["group_offsets"], res[1]["group_offsets"][1:] + S0]).astype(np.int32)
    z = cat([res[0]["z"], res[1]["z"]])
    ids, mask = cat([res[0]["ids"], res[1]["ids"]]), cat([res[0]["mask"], res[1]["mask"]])
    op = oracle_params(__import__("paper_2607_24062_gb300").Params())
    ref = O.step(z, ids, mask, cat([res[0]["mu"], res[1]["mu"]]), cat([res[0]["R"], res[1]["R"]]), so, go, op)
    coef = O.loss_coefficients(ref.weight, ref.adv, mask, so, ref.seq, ref.grp, ref.batch, op)
    for r, sl in ((0, slice(0, T0)), (1, slice(T0, None))):
        assert_close_rel(res[r]["X"], ref.state.X, floor=1e-12, what=f"X (rank {r})")
        assert_close_rel(res[r]["weight"], ref.weight[sl], floor=1e-7, what=f"weight (rank {r})")
        assert_close_rel(res[r]["coef"], coef[sl], floor=1e-12, what=f"coef (rank {r})")
    # without the exchange each rank would calibrate X on its own prompts
    lone = O.step(res[0]["z"], res[0]["ids"], res[0]["mask"], res[0]["mu"], res[0]["R"], res[0]["seq_offsets"],
                  res[0]["group_offsets"], op)
    assert lone.state.X != pytest.approx(ref.state.X, rel=1e-6)
