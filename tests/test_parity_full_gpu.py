"""GPU parity at the full workload sizes, in the launch configuration the
benchmark times.  The vocabulary-wide outputs (lse, logp, entropy, gradient)
are checked element by element on sampled rows: 4,096 random valid rows,
every row of 4 whole responses, the first and last row of the batch, and the
first and last row of each gradient chunk.  Every O(T) output is checked on
all rows, stage-isolated: the oracle's discrepancy, advantage and controller
stages are fed the GPU's fp32 log-probs.  The oracle's own full chain (its
log-softmax, then the discrepancy) is checked on the whole responses."""

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from parity import (VocabRowCheck, assert_close_abs, assert_close_rel, assert_grad_rows, assert_loss, compare_batch,
                    compare_grp, compare_seq, grad_rows, host, oracle_params)

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import api  # noqa: E402

DEV = "cuda"


def _sample_rows(b, rng, n_random=4096, n_whole=4, extra=()):
    mask = host(b.mask)
    so = host(b.seq_offsets)
    valid = np.flatnonzero(mask)
    rows = set(rng.choice(valid, size=min(n_random, len(valid)), replace=False).tolist())
    whole = rng.choice(b.S, size=n_whole, replace=False) if n_whole else np.zeros(0, dtype=np.int64)
    for i in whole:
        rows.update(range(int(so[i]), int(so[i + 1])))
    rows.update([0, b.T - 1, *extra])
    return np.array(sorted(rows)), whole


def _oracle_O_T(step, b, op):
    """Stage-isolated O(T) stages on the GPU's log-probs, compared with the GPU."""
    lp = host(step.logp).astype(np.float64)
    Hh = host(step.entropy).astype(np.float64)
    mask, so, go = host(b.mask), host(b.seq_offsets), host(b.group_offsets)
    mu = host(b.logp_mu).astype(np.float64)
    lr, d, seq, grp, batch, f = O.seq_discrepancy(lp, mu, mask, so, go, Hh)
    assert f == 0
    assert_close_abs(host(step.disc.lr), lr, 1e-6 * np.maximum(1.0, np.abs(lr)), "lr")
    assert_close_rel(host(step.disc.d), d, floor=1e-9, what="d")
    compare_seq(step.seq_host(), seq)
    compare_grp(step.grp_host(), grp)
    gb = step.batch_host()
    compare_batch(gb, batch)
    adv = O.grpo_advantage(host(b.rewards).astype(np.float64), go, op)
    assert_close_rel(host(step.adv), adv, floor=1e-6, what="adv")
    w, alpha, st, info, f = O.controller_step(O.controller_init(op), op, lr, mask, so, go, seq, grp, batch, adv)
    gst = step.state_host()
    assert_close_rel(gst["X"], st.X, floor=1e-12, what="X")
    assert_close_rel(host(step.alpha), alpha, floor=1e-6, what="alpha")
    assert_close_rel(host(step.weight), w, floor=1e-7, what="weight")
    assert_close_rel(gb["w_mean"], info["w_mean"], floor=1e-9, what="w_mean")
    assert_close_rel(gb["trunc_frac"], info["trunc_frac"], floor=2.0 / batch["n_tokens"], what="trunc_frac")
    coef = O.loss_coefficients(w, adv, mask, so, seq, grp, batch, op)
    assert_close_rel(host(step.coef), coef, floor=1e-12, what="coef")
    tl, loss = O.surrogate_loss(lp, None, adv, w, mask, so, seq, grp, batch, op)
    assert_close_rel(host(step.token_loss), tl, floor=1e-12, what="token_loss")
    assert_loss(float(step.loss), loss, tl)
    return dict(lr=lr, seq=seq, grp=grp, batch=batch, adv=adv, w=w, coef=coef)


def _check_rows(step, b, rows, ref, op):
    """a1 and a6 on `rows` against the oracle's own fp64 log-softmax and gradient (blocks of rows in the oracle
    pool); returns the checker, which keeps the oracle's logp and entropy of those rows."""
    chk = VocabRowCheck(b.T, host(b.ids), host(b.mask), host(b.seq_offsets), ref, op)
    chk.submit(b.logits, b.V, rows, step.lse, step.logp, step.entropy, step.grad)
    assert chk.finish() == len(rows)
    return chk


def _oracle_chain_on_whole(step, b, whole, chk):
    """The oracle's own chain (its log-softmax, then the discrepancy) on whole responses; the oracle's log-probs
    and entropies are those the row check computed."""
    so, mask = host(b.seq_offsets), host(b.mask)
    mu = host(b.logp_mu).astype(np.float64)
    gseq = step.seq_host()
    for i in whole:
        r = np.arange(int(so[i]), int(so[i + 1]))
        ologp = np.array([chk.oracle_logp[t] for t in r.tolist()])
        oH = np.array([chk.oracle_entropy[t] for t in r.tolist()])
        lr, d, seq, _, _, _ = O.seq_discrepancy(ologp, mu[r], mask[r], [0, len(r)], [0, 1], oH)
        assert int(gseq["n"][i]) == int(seq["n"][0])
        assert_close_rel(gseq["mean_d"][i], seq["mean_d"][0], floor=1e-7, what=f"D_{i} (oracle chain)")
        assert_close_abs(gseq["sum_lr"][i], seq["sum_lr"][0], 1e-3 * max(1.0, abs(seq["sum_lr"][0])),
                         what=f"S_{i} (oracle chain)")


@pytest.mark.parametrize("name", ["grpo", "qwen"])
def test_full_size_workload(name):
    torch.cuda.empty_cache()
    spec = W.SPECS[name]
    b = W.generate(spec, device=DEV)
    p = acrl.Params()
    op = oracle_params(p)
    step = acrl.AcrlStep.for_batch(b, p)
    step.run_batch(b)
    torch.cuda.synchronize()
    assert api.read_flags(step.flags) == 0
    ref = _oracle_O_T(step, b, op)
    rng = np.random.default_rng(11)
    rows, whole = _sample_rows(b, rng)
    chk = _check_rows(step, b, rows, ref, op)
    _oracle_chain_on_whole(step, b, whole, chk)
    # cached-old path (lse recomputed inside the gradient call by a first sweep over each row) on the first
    # 4,096 rows: the same gradient as the streaming call
    R = min(4096, b.T)
    g2, tl2, _ = api.loss_grad_logits(b.logits[:R], b.ids[:R], b.mask[:R], None, step.logp[:R], step.coef[:R],
                                      p.clip_eps, V=b.V)
    torch.cuda.synchronize()
    rr = np.arange(0, R, 7)
    ref = grad_rows(step.grad, rr, b.V)
    assert_grad_rows(grad_rows(g2, rr, b.V), ref, np.abs(host(step.coef)[rr]) + 1e-30, host(b.ids)[rr],
                     what="grad (lse recomputed)")
    assert_close_rel(host(tl2), host(step.token_loss)[:R], rel=1e-4, floor=1e-12, what="token_loss (lse recomputed)")
    # masked rows: zero gradient and zero statistics
    masked = np.flatnonzero(host(b.mask) == 0)
    if len(masked):
        mr = masked[:: max(1, len(masked) // 64)]
        assert np.all(grad_rows(step.grad, mr, b.V) == 0)
        assert np.all(host(step.logp)[mr] == 0) and np.all(host(step.entropy)[mr] == 0)
    # the whole step again from a fresh controller: every output bit for bit the same (fixed reduction orders,
    # no atomics)
    del g2, tl2
    step2 = acrl.AcrlStep.for_batch(b, p)
    step2.run_batch(b)
    torch.cuda.synchronize()
    for name in ("lse", "logp", "entropy", "weight", "coef", "alpha", "adv", "token_loss", "loss", "state"):
        assert torch.equal(getattr(step, name), getattr(step2, name)), name
    assert torch.equal(step.disc.batch, step2.disc.batch) and torch.equal(step.disc.seq, step2.disc.seq)
    for r0 in range(0, b.T, 8192):
        r1 = min(b.T, r0 + 8192)
        assert torch.equal(step.grad[r0:r1].view(torch.int16), step2.grad[r0:r1].view(torch.int16)), (r0, r1)


def test_long_workload_chunked():
    """~328k rows at V = 151,936: the logits stay resident (99.6 GB) and the
    gradient goes through a reused 65,536-row chunk buffer; each chunk is
    checked on sampled rows as it is produced."""
    torch.cuda.empty_cache()
    spec = W.LONG
    b = W.generate(spec, device=DEV)
    p = acrl.Params()
    op = oracle_params(p)
    step = acrl.AcrlStep.for_batch(b, p, grad_rows=spec.chunk_rows)
    step.statistics(b.logits, b.ids, b.mask, b.logp_mu, b.rewards, b.seq_offsets, b.group_offsets)
    torch.cuda.synchronize()
    lp = host(step.logp).astype(np.float64)
    mask, so, go = host(b.mask), host(b.seq_offsets), host(b.group_offsets)
    mu = host(b.logp_mu).astype(np.float64)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(lp, mu, mask, so, go, host(step.entropy).astype(np.float64))
    compare_seq(step.seq_host(), seq)
    compare_grp(step.grp_host(), grp)
    compare_batch(step.batch_host(), batch)
    adv = O.grpo_advantage(host(b.rewards).astype(np.float64), go, op)
    w, alpha, st, info, _ = O.controller_step(O.controller_init(op), op, lr, mask, so, go, seq, grp, batch, adv)
    assert_close_rel(host(step.weight), w, floor=1e-7, what="weight")
    coef = O.loss_coefficients(w, adv, mask, so, seq, grp, batch, op)
    assert_close_rel(host(step.coef), coef, floor=1e-12, what="coef")
    ref = dict(seq=seq, grp=grp, batch=batch, adv=adv, w=w, coef=coef)
    rng = np.random.default_rng(5)
    rows_all, whole = _sample_rows(b, rng)
    chk = VocabRowCheck(b.T, host(b.ids), mask, so, ref, op)
    checked = []

    def on_chunk(r0, r1, g):
        # the chunk buffer is reused for the next chunk: the rows are copied out before this returns
        torch.cuda.synchronize()
        rows = rows_all[(rows_all >= r0) & (rows_all < r1)]
        rows = np.unique(np.concatenate([rows, [r0, r1 - 1]]))
        chk.submit(b.logits, b.V, rows, step.lse, step.logp, step.entropy, grad=g, grad_row0=r0)
        checked.append(len(rows))

    step.gradient(b.logits, b.ids, b.mask, chunk_rows=spec.chunk_rows, on_chunk=on_chunk)
    torch.cuda.synchronize()
    assert chk.finish() == sum(checked) >= len(rows_all)
    assert len(checked) == (b.T + spec.chunk_rows - 1) // spec.chunk_rows
    _oracle_chain_on_whole(step, b, whole, chk)
    tl, loss = O.surrogate_loss(lp, None, adv, w, mask, so, seq, grp, batch, op)
    assert_close_rel(host(step.token_loss), tl, floor=1e-12, what="token_loss")
    assert_loss(float(step.loss), loss, tl)
    assert api.read_flags(step.flags) == 0
