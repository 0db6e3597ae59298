"""Multi-rank path on CPU with the gloo backend (world size 2).

Each rank owns whole prompts; the ranks sum three fields of their batch
statistics (distributed.allreduce_batch_stats) before the controller.  The
result must equal the single-process oracle on the concatenated batch: one
global X (Sec. 4.1's mean over all prompts) and the loss normalised by the
global prompt count.  A rank that dies before the exchange must surface as an
error on the surviving rank, not as a hang."""

import datetime
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle as O
import workloads as W
from paper_2607_24062_gb300 import _abi
from paper_2607_24062_gb300 import distributed as D

SPEC = W.small_variant(W.LONG, name="dist", n_prompts=3, group_size=4, len_lo=20, len_hi=120, perturb_frac=0.3,
                       perturb_std=0.3)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _shard(seed):
    d = W.token_level(SPEC, seed)
    return {k: (v.numpy() if isinstance(v, torch.Tensor) else v) for k, v in d.items()}


def _encode(b):
    arr = np.zeros(1, dtype=_abi.BATCH_DTYPE)
    for k in arr.dtype.names:
        if k in b:
            arr[k] = b[k]
    return torch.from_numpy(arr.view(np.uint8).copy())


def _decode(buf):
    return buf.numpy().view(_abi.BATCH_DTYPE)[0]


def _rank_result(d, batch_override, p):
    so, go, mask = d["seq_offsets"], d["group_offsets"], d["mask"]
    lr, dd, seq, grp, batch, _ = O.seq_discrepancy(d["logp_pi"].astype(np.float64), d["logp_mu"].astype(np.float64),
                                                   mask, so, go)
    if batch_override is not None:
        batch = batch_override(batch)
    adv = O.grpo_advantage(d["rewards"].astype(np.float64), go, p)
    w, alpha, st, info, _ = O.controller_step(O.controller_init(p), p, lr, mask, so, go, seq, grp, batch, adv)
    coef = O.loss_coefficients(w, adv, mask, so, seq, grp, batch, p)
    return st.X, w, coef


def _worker(rank, world, port, shards, results):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    p = O.Params()

    def exchange(batch):
        buf = _encode(batch)
        D.allreduce_batch_stats(buf)
        g = _decode(buf)
        out = dict(batch)
        out["n_tokens"] = int(g["n_tokens"])
        out["n_groups_valid"] = int(g["n_groups_valid"])
        out["Y_sum"] = float(g["Y_sum"])
        out["Y_mean"] = out["Y_sum"] / out["n_groups_valid"]
        return out

    X, w, coef = _rank_result(shards[rank], exchange, p)
    results[rank] = (X, w, coef)
    dist.destroy_process_group()


def _concat(shards):
    out = {}
    T0, S0 = 0, 0
    so, go = [np.array([0])], [np.array([0], dtype=np.int32)]
    for d in shards:
        so.append(d["seq_offsets"][1:] + T0)
        go.append(d["group_offsets"][1:] + S0)
        T0 += d["T"]
        S0 += len(d["seq_offsets"]) - 1
    for k in ("logp_pi", "logp_mu", "mask", "rewards"):
        out[k] = np.concatenate([d[k] for d in shards])
    out["seq_offsets"] = np.concatenate(so)
    out["group_offsets"] = np.concatenate(go).astype(np.int32)
    return out


def test_sharded_calibration_equals_unsharded():
    shards = [_shard(D.shard_seed(11, r)) for r in range(2)]
    with mp.get_context("spawn").Manager() as mgr:
        results = mgr.dict()
        mp.start_processes(_worker, args=(2, _free_port(), shards, results), nprocs=2, start_method="spawn")
        res = dict(results)
    X_all, w_all, coef_all = _rank_result(_concat(shards), None, O.Params())
    assert res[0][0] == pytest.approx(X_all, rel=1e-12) and res[1][0] == pytest.approx(X_all, rel=1e-12)
    T0 = shards[0]["T"]
    np.testing.assert_allclose(np.concatenate([res[0][1], res[1][1]]), w_all, rtol=1e-12)
    np.testing.assert_allclose(np.concatenate([res[0][2], res[1][2]]), coef_all, rtol=1e-12, atol=1e-300)
    # without the exchange a rank would calibrate on its own prompts only
    X_local, _, _ = _rank_result(shards[0], None, O.Params())
    assert X_local != pytest.approx(X_all, rel=1e-6)
    assert len(res[0][1]) == T0


def _dying_worker(rank, world, port, results):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=5))
    if rank == 1:
        os._exit(0)          # leaves between steps, before the exchange, without a collective in flight
    buf = _encode({"n_tokens": 10, "n_groups_valid": 2, "Y_sum": 0.03})
    try:
        D.allreduce_batch_stats(buf)
        results[0] = "completed"
    except Exception as e:  # the surviving rank learns of it from the process group
        results[0] = f"error: {type(e).__name__}"


def test_dead_rank_surfaces_as_error():
    with mp.get_context("spawn").Manager() as mgr:
        results = mgr.dict()
        ctx = mp.start_processes(_dying_worker, args=(2, _free_port(), results), nprocs=2, start_method="spawn",
                                 join=False)
        for p in ctx.processes:
            p.join(timeout=60)
        alive = [p.is_alive() for p in ctx.processes]
        for p in ctx.processes:
            if p.is_alive():
                p.kill()
        assert not any(alive), "a rank hung"
        assert str(results.get(0, "")).startswith("error"), results.get(0)
