"""More token rows than a 32-bit index holds (T = 2^31 + 3, V = 8), through
every per-token call, so that each per-token array is addressed beyond
2^31 elements.  The oracle checks sampled rows one by one; the rest is
checked through properties that hold at any size:

- a row of zeros is uniform: lse = ln 8, log p = -ln 8, H = ln 8;
- dL/dlogits = coef (p - onehot) on the planted rows, -coef as the on-policy
  token loss on every row and their sum as the loss;
- with mu = pi the discrepancy is 0 everywhere, every ACRL weight is 1, the
  counts are exact and coef_t = A_i / (Q_eff G_g n_i), with the advantages
  the oracle's.
Peak device memory is about 120 GB (the bf16 logits and gradient are 34 GB
each)."""

import math

import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import api  # noqa: E402

T = (1 << 31) + 3
V = 8


def _sample(rng, n=2000):
    edge = np.array([0, 1, (1 << 31) - 2, (1 << 31) - 1, 1 << 31, (1 << 31) + 1, T - 1], dtype=np.int64)
    return np.unique(np.concatenate([edge, rng.integers(0, T, size=n)]))


def test_rows_beyond_32_bit_indices():
    dev = torch.device("cuda")
    torch.cuda.empty_cache()
    rng = np.random.default_rng(5)
    planted = np.array([0, (1 << 31) - 1, 1 << 31, T - 1], dtype=np.int64)
    zp = rng.normal(0.0, 2.0, size=(len(planted), V))
    zp_bf16 = torch.tensor(zp, dtype=torch.float32).to(torch.bfloat16)
    zp = zp_bf16.to(torch.float64).numpy()
    ids_p = rng.integers(0, V, size=len(planted)).astype(np.int32)

    logits = torch.zeros((T, V), dtype=torch.bfloat16, device=dev)
    ids = torch.zeros(T, dtype=torch.int32, device=dev)
    pidx = torch.as_tensor(planted, device=dev)
    logits[pidx] = zp_bf16.to(dev)
    ids[pidx] = torch.as_tensor(ids_p, device=dev)
    flags = api.new_flags(dev)
    lse, logp, H = api.token_stats(logits, ids, None, V=V, flags=flags)

    lnV = math.log(V)
    rows = np.setdiff1d(_sample(rng), planted)
    ridx = torch.as_tensor(rows, device=dev)
    for t_out, want in ((lse, lnV), (logp, -lnV), (H, lnV)):
        np.testing.assert_allclose(t_out[ridx].cpu().numpy(), want, atol=2e-5)
    olse, ologp, oH, _ = O.token_stats(zp, ids_p, None)
    np.testing.assert_allclose(lse[pidx].cpu().numpy(), olse, atol=2e-4)
    np.testing.assert_allclose(logp[pidx].cpu().numpy(), ologp, atol=2e-4)
    np.testing.assert_allclose(H[pidx].cpu().numpy(), oH, rtol=1e-3, atol=1e-5)

    coef = torch.full((T,), 0.5, dtype=torch.float32, device=dev)
    del H
    grad, token_loss, loss = api.loss_grad_logits(logits, ids, None, lse, None, coef, 0.2, V=V, flags=flags)
    assert api.read_flags(flags) == 0
    p = np.exp(zp - olse[:, None])
    want = 0.5 * (p - np.eye(V)[ids_p])
    np.testing.assert_allclose(grad[pidx].double().cpu().numpy(), want, rtol=1e-2, atol=1e-6)
    g0 = grad[torch.as_tensor(rows[:64], device=dev)].double().cpu().numpy()
    np.testing.assert_allclose(g0, np.tile(0.5 * (np.full(V, 1.0 / V) - np.eye(V)[0]), (64, 1)), rtol=1e-2)
    np.testing.assert_allclose(token_loss[ridx].cpu().numpy(), -0.5, rtol=1e-6)
    np.testing.assert_allclose(token_loss[pidx].cpu().numpy(), -0.5, rtol=1e-6)
    assert float(loss) == pytest.approx(-0.5 * T, rel=1e-6)
    del logits, grad, token_loss, coef, lse, ids
    torch.cuda.empty_cache()

    # the O(T) calls: 16,384 prompts x 8 responses of 16,384 tokens (the last one 3 more)
    lp = torch.full((T,), -lnV, dtype=torch.float32, device=dev)
    del logp
    torch.cuda.empty_cache()
    S, G = 1 << 17, 8
    Gn = S // G
    cuts = np.arange(S + 1, dtype=np.int64) * 16384
    cuts[-1] = T
    so = torch.as_tensor(cuts, device=dev)
    go = torch.as_tensor(np.arange(Gn + 1, dtype=np.int32) * G, device=dev)
    R = (np.arange(S) % 3 == 0).astype(np.float32)
    prm = acrl.Params(X_init=0.1)
    disc = api.seq_discrepancy(lp, lp, None, so, go, flags=flags)
    adv = api.grpo_advantage(torch.as_tensor(R, device=dev), go, prm, flags=flags)
    w, coef, alpha = api.controller_step(api.controller_init(prm), prm, disc, None, so, go, adv, flags=flags)
    assert api.read_flags(flags) == 0
    seq, grp, batch = disc.seq_host(), disc.grp_host(), disc.batch_host()
    n = np.diff(cuts)
    assert np.array_equal(seq["n"], n) and int(batch["n_tokens"]) == T
    assert int(batch["n_groups_valid"]) == Gn and np.all(grp["Y"] == 0.0)
    assert float(batch["d_max"]) == 0.0
    sidx = torch.as_tensor(_sample(rng), device=dev)
    assert torch.all(disc.lr[sidx] == 0) and torch.all(disc.d[sidx] == 0) and torch.all(w[sidx] == 1.0)
    A = O.grpo_advantage(R.astype(np.float64), np.arange(Gn + 1) * G, O.Params())
    np.testing.assert_allclose(adv.cpu().numpy(), A, rtol=1e-6, atol=1e-7)
    rows = _sample(rng)
    resp = np.searchsorted(cuts, rows, side="right") - 1
    want = A[resp] / (Gn * G * n[resp])
    np.testing.assert_allclose(coef[torch.as_tensor(rows, device=dev)].cpu().numpy(), want, rtol=1e-5, atol=0)
