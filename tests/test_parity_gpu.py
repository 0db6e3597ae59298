"""GPU parity: the CUDA path, called through the C ABI, against the float64
oracle on the same seeded inputs.  Small shapes are compared element by
element over the whole chain; the full-size workloads on sampled rows plus
every O(T) output."""

import math
import os

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from parity import (TOL_LOGP, assert_close_abs, assert_close_rel, assert_grad_rows, assert_loss, compare_batch,
                    compare_grp, compare_seq, grad_rows, host, oracle_params, rows_f64)

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import api  # noqa: E402

DEV = "cuda"


def _gen(spec, seed=None, mutate=None):
    b = W.generate(spec, seed=seed, device=DEV)
    if mutate:
        mutate(b)
    return b


def _host_inputs(b):
    return dict(ids=host(b.ids), mask=host(b.mask), mu=host(b.logp_mu).astype(np.float64),
                R=host(b.rewards).astype(np.float64), so=host(b.seq_offsets), go=host(b.group_offsets))


def _full_chain_check(b, params, state=None):
    """Run the GPU step and the oracle step on every row; compare everything."""
    step = acrl.AcrlStep.for_batch(b, params)
    if state is not None:
        step.state.copy_(state)
    step.run_batch(b)
    torch.cuda.synchronize()
    h = _host_inputs(b)
    op = oracle_params(params)
    z = rows_f64(b.logits, np.arange(b.T), b.V)
    ostate = None
    if state is not None:
        s = api.read_structs(state, api.STATE_DTYPE, 1)[0]
        ostate = O.ControllerState(X=float(s["X"]), calib_sum=float(s["calib_sum"]),
                                   calib_count=int(s["calib_count"]), calib_done_steps=int(s["calib_done"]),
                                   step=int(s["step"]), calibrated=bool(s["calibrated"]))
    res = O.step(z, h["ids"], h["mask"], h["mu"], h["R"], h["so"], h["go"], op, state=ostate)
    # a1
    assert_close_abs(host(step.logp), res.logp, TOL_LOGP, "logp")
    assert_close_abs(host(step.lse), res.lse, TOL_LOGP, "lse")
    assert_close_rel(host(step.entropy), res.H, floor=1e-5, what="entropy")
    # a2/a3: against the fp64 chain, d inherits the log-prob bar: |dd| <= pi |dlogp|
    assert_close_abs(host(step.disc.lr), res.lr, TOL_LOGP, "lr")
    assert_close_rel(host(step.disc.d), res.d, floor=TOL_LOGP * np.exp(res.logp), what="d")
    _stage_isolated_discrepancy(step, h)
    compare_seq(step.seq_host(), res.seq)
    compare_grp(step.grp_host(), res.grp)
    gb = step.batch_host()
    compare_batch(gb, res.batch)
    # a4
    assert_close_rel(host(step.adv), res.adv, floor=1e-6, what="adv")
    # a5
    st = step.state_host()
    assert bool(st["calibrated"]) == res.state.calibrated and int(st["step"]) == res.state.step
    assert_close_rel(st["X"], res.state.X, floor=1e-12, what="X")
    assert_close_rel(gb["X"], res.info["X"] if res.state.calibrated else 0.0, floor=1e-12, what="batch.X")
    assert_close_rel(host(step.alpha), res.alpha, floor=1e-6, what="alpha")
    assert_close_rel(host(step.weight), res.weight, floor=1e-7, what="weight")
    assert_close_rel(gb["w_mean"], res.info["w_mean"], floor=1e-9, what="w_mean")
    assert_close_rel(gb["trunc_frac"], res.info["trunc_frac"], floor=2.0 / max(1, res.batch["n_tokens"]),
                     what="trunc_frac")
    coef_ref = O.loss_coefficients(res.weight, res.adv, h["mask"], h["so"], res.seq, res.grp, res.batch, op)
    assert_close_rel(host(step.coef), coef_ref, floor=1e-12, what="coef")
    # a6
    assert_close_rel(host(step.token_loss), res.token_loss, floor=1e-12, what="token_loss")
    assert_loss(float(step.loss), res.loss, res.token_loss)
    assert_grad_rows(grad_rows(step.grad, np.arange(b.T), b.V), res.grad, coef_ref, h["ids"],
                     row_floor=1e-6 if op.entropy_coeff else 0.0)
    flags = api.read_flags(step.flags)
    assert flags == res.flags, (flags, res.flags)
    return step, res


def _stage_isolated_discrepancy(step, h):
    """K2's own arithmetic: the oracle fed the GPU's fp32 log-probs."""
    lp = host(step.logp).astype(np.float64)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(lp, h["mu"], h["mask"], h["so"], h["go"],
                                                  host(step.entropy).astype(np.float64))
    assert_close_abs(host(step.disc.lr), lr, 1e-6 * np.maximum(1.0, np.abs(lr)), "lr (isolated)")
    assert_close_rel(host(step.disc.d), d, floor=1e-9, what="d (isolated)")
    compare_seq(step.seq_host(), seq, "seq (isolated)")
    compare_grp(step.grp_host(), grp, "grp (isolated)")
    compare_batch(step.batch_host(), batch, "batch (isolated)")
    return lr, d, seq, grp, batch


SMALL = {
    "tiny": W.TINY,
    "ragged_warp": W.small_variant(W.GRPO, name="ragged_warp", n_prompts=3, group_size=4, len_lo=1, len_hi=90,
                                   V=5003, pad_multiple=16, ld_pad=8),
    "ragged_cta": W.small_variant(W.QWEN, name="ragged_cta", n_prompts=2, group_size=3, len_lo=3, len_hi=40,
                                  V=20011, ld_pad=24),
    "qwen_vocab": W.small_variant(W.QWEN, name="qwen_vocab", n_prompts=2, group_size=4, len_lo=8, len_hi=24),
    # degenerate and wide vocabularies: one token (logp = 0, H = 0, zero gradient), and 2^18 + 3 columns
    "one_token_vocab": W.small_variant(W.GRPO, name="one_token_vocab", n_prompts=2, group_size=3, len_lo=5,
                                       len_hi=30, V=1),
    "wide_vocab": W.small_variant(W.QWEN, name="wide_vocab", n_prompts=2, group_size=2, len_lo=8, len_hi=40,
                                  V=262147),
}


@pytest.mark.parametrize("name", list(SMALL))
def test_full_chain_small(name):
    _full_chain_check(_gen(SMALL[name], seed=123), acrl.Params())


def _empty_seq(b):
    # response 1 fully masked, and its prompt's other members keep going
    so = host(b.seq_offsets)
    b.mask[int(so[1]):int(so[2])] = 0


def test_empty_sequence_and_group():
    spec = W.small_variant(W.GRPO, name="empties", n_prompts=3, group_size=2, len_lo=5, len_hi=50, V=3001)

    def mutate(b):
        so = host(b.seq_offsets)
        b.mask[int(so[1]):int(so[2])] = 0          # one empty response
        b.mask[int(so[4]):int(so[6])] = 0          # a whole empty prompt

    step, res = _full_chain_check(_gen(spec, seed=9, mutate=mutate), acrl.Params())
    assert res.batch["n_groups_valid"] == 2


# the granularity of Y only matters for the modes that compare Y with X
_MODE_CASES = [(m, acrl.Y_GROUP) for m in (acrl.MODE_NONE, acrl.MODE_TIS, acrl.MODE_MIS, acrl.MODE_ACRL_CONTINUOUS)] + \
    [(m, y) for m in (acrl.MODE_ACRL, acrl.MODE_ACRL_FALLBACK) for y in (acrl.Y_GROUP, acrl.Y_SEQUENCE, acrl.Y_BATCH)]


@pytest.mark.parametrize("mode,y_gran", _MODE_CASES)
def test_modes(mode, y_gran):
    spec = W.small_variant(W.QWEN, name="modes", n_prompts=3, group_size=4, len_lo=4, len_hi=60, V=2048,
                           perturb_frac=0.5, perturb_std=0.3)
    _full_chain_check(_gen(spec, seed=77), acrl.Params(mode=mode, y_gran=y_gran, gamma=1.3, C=5.0))


@pytest.mark.parametrize("kw", [dict(agg=acrl.AGG_TOKEN_MEAN), dict(adv_ddof=0), dict(adv_eps=0.0), dict(X_init=0.013),
                                dict(singleton_rule=acrl.SINGLETON_ZERO), dict(calib_steps=2),
                                dict(entropy_coeff=0.001), dict(entropy_coeff=0.05, agg=acrl.AGG_TOKEN_MEAN),
                                dict(X_init=0.013, x_ema=0.3), dict(mode=acrl.MODE_ACRL_CONTINUOUS, kappa=3.0)])
def test_param_options(kw):
    spec = W.small_variant(W.TINY, name="opts", n_prompts=3, group_size=2, len_lo=20, len_hi=70, V=1000)
    _full_chain_check(_gen(spec, seed=5), acrl.Params(**kw))


def test_singletons_tiny_grpo_rule():
    # tiny workload: 4 prompts with one response each; A = R under MEAN0_STD1
    step, res = _full_chain_check(_gen(W.TINY), acrl.Params())
    np.testing.assert_array_equal(host(step.adv), host(W.generate(W.TINY, device="cpu").rewards))


def test_uniform_logits_and_equal_policies():
    # uniform logits: logp = -ln V and H = ln V; mu = pi: lr = d = 0, every weight 1, X -> 0 (flagged)
    T, V = 12, 151936
    logits = torch.full((T, V), 0.5, dtype=torch.bfloat16, device=DEV)
    ids = torch.randint(0, V, (T,), dtype=torch.int32, device=DEV)
    lse, logp, H = api.token_stats(logits, ids, None, V=V)
    assert_close_abs(host(logp), -math.log(V), 1e-5, "uniform logp")
    assert_close_rel(host(H), math.log(V), rel=1e-5, what="uniform entropy")
    so = torch.tensor([0, 4, 8, 12], dtype=torch.int64, device=DEV)
    go = torch.tensor([0, 2, 3], dtype=torch.int32, device=DEV)
    p = acrl.Params()
    flags = api.new_flags()
    disc = api.seq_discrepancy(logp, logp.clone(), None, so, go, H, flags=flags)
    adv = api.grpo_advantage(torch.tensor([1.0, 0.0, 1.0], device=DEV), go, p, flags=flags)
    state = api.controller_init(p)
    w, coef, alpha = api.controller_step(state, p, disc, None, so, go, adv, flags=flags)
    assert torch.all(disc.lr == 0) and torch.all(disc.d == 0)
    assert torch.all(w == 1.0) and torch.all(alpha == 0.0)
    assert float(api.read_state(state)["X"]) == 0.0
    assert api.read_flags(flags) == acrl.FLAG_X_NONPOS


@pytest.mark.parametrize("beta", [0.0, 0.01])
@pytest.mark.parametrize("V", [20011, 4099, 32000, 49152, 151936])
def test_old_logp_and_recomputed_lse(V, beta):
    """Cached-old path: weights from old log-probs, LSE recomputed in the gradient kernel, r != 1 with clipping
    (warp row teams, and CTAs of 128, 256 and 512 threads; rows held whole in shared memory between the two
    sweeps, and rows of which the first 96 KB are held there, 128 KB more in tensor memory and the rest read
    again from L2; with and without the entropy bonus)."""
    spec = W.small_variant(W.QWEN, name="offpolicy", n_prompts=2, group_size=4, len_lo=10, len_hi=80, V=V)
    b = _gen(spec, seed=31)
    p = acrl.Params(entropy_coeff=beta)
    gen = torch.Generator(device=DEV).manual_seed(3)
    lse, logp, H = api.token_stats(b.logits, b.ids, b.mask, V=b.V)
    old = (logp + 0.3 * torch.randn(b.T, generator=gen, device=DEV)).clamp(max=0.0)
    disc = api.seq_discrepancy(old, b.logp_mu, b.mask, b.seq_offsets, b.group_offsets, H)
    adv = api.grpo_advantage(b.rewards, b.group_offsets, p)
    state = api.controller_init(p)
    ent_coef = torch.empty(b.T, device=DEV) if beta else None
    w, coef, alpha = api.controller_step(state, p, disc, b.mask, b.seq_offsets, b.group_offsets, adv,
                                         ent_coef=ent_coef)
    for recompute in (False, True):
        grad, tl, loss = api.loss_grad_logits(b.logits, b.ids, b.mask, None if recompute else lse, old, coef,
                                              p.clip_eps, V=b.V, entropy=H if beta else None, ent_coef=ent_coef)
        torch.cuda.synchronize()
        h = _host_inputs(b)
        op = oracle_params(p)
        z = rows_f64(b.logits, np.arange(b.T), b.V)
        olse, ologp, oH, _ = O.token_stats(z, h["ids"], h["mask"])
        oold = host(old).astype(np.float64)
        lr, d, seq, grp, batch, _ = O.seq_discrepancy(oold, h["mu"], h["mask"], h["so"], h["go"], oH)
        oadv = O.grpo_advantage(h["R"], h["go"], op)
        ow, oalpha, ost, info, _ = O.controller_step(O.controller_init(op), op, lr, h["mask"], h["so"], h["go"], seq,
                                                     grp, batch, oadv)
        assert_close_rel(host(w), ow, floor=1e-7, what="weight")
        ograd, otl, oloss = O.loss_grad_logits(z, h["ids"], h["mask"], None, oold, oadv, ow, h["so"], seq, grp,
                                               batch, op)
        coef_ref = O.loss_coefficients(ow, oadv, h["mask"], h["so"], seq, grp, batch, op)
        if beta:
            ecoef = O.entropy_coefficients(h["mask"], h["so"], seq, grp, batch, op)
            assert_close_rel(host(ent_coef), ecoef, floor=1e-12, what="ent_coef")
        r = np.exp(ologp - oold)
        gate = np.where(coef_ref >= 0, r <= 1 + op.clip_eps, r >= 1 - op.clip_eps)
        assert 0 < gate.sum() < len(gate)   # both branches exercised
        # the sampled column's absolute floor scales with the largest coefficient on the row
        scale = np.abs(coef_ref * r * gate) + (ecoef * (1 + np.abs(oH)) if beta else 0.0)
        assert_grad_rows(grad_rows(grad, np.arange(b.T), b.V), ograd, scale, h["ids"], row_floor=1e-6 if beta else 0)
        assert_close_rel(host(tl), otl, floor=1e-12, what="token_loss")
        assert_loss(float(loss), oloss, otl)


@pytest.mark.parametrize("V", [4099, 20011, 32000, 49152, 151936])
def test_gradient_undefined_rows_on_gpu(V):
    """Readings c17 and c18 in the gradient call: a live row with a NaN or an
    infinite logit, or with a NaN old log-prob, gets a NaN gradient row and a
    NaN token loss and the call raises NONFINITE, whether the lse is given
    (from the statistics call, NaN there too) or recomputed; a row whose
    coefficient is 0 stays a zero row with token loss 0 whatever its logits
    hold; every other row matches the oracle element by element."""
    spec = W.small_variant(W.QWEN, name="undefined", n_prompts=2, group_size=4, len_lo=10, len_hi=40, V=V)
    b = _gen(spec, seed=37)
    p = acrl.Params()
    op = oracle_params(p)
    h = _host_inputs(b)
    lse0, logp0, H0 = api.token_stats(b.logits, b.ids, b.mask, V=b.V)
    gen = torch.Generator(device=DEV).manual_seed(5)
    old = (logp0 + 0.1 * torch.randn(b.T, generator=gen, device=DEV)).clamp(max=0.0)
    disc = api.seq_discrepancy(old, b.logp_mu, b.mask, b.seq_offsets, b.group_offsets, H0)
    adv = api.grpo_advantage(b.rewards, b.group_offsets, p)
    w, coef, alpha = api.controller_step(api.controller_init(p), p, disc, b.mask, b.seq_offsets, b.group_offsets, adv)
    torch.cuda.synchronize()
    # the oracle's weights from the same (clean) inputs
    z0 = rows_f64(b.logits, np.arange(b.T), b.V)
    _, ologp0, oH0, _ = O.token_stats(z0, h["ids"], h["mask"])
    oold_clean = host(old).astype(np.float64)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(oold_clean, h["mu"], h["mask"], h["so"], h["go"], oH0)
    oadv = O.grpo_advantage(h["R"], h["go"], op)
    ow, _, _, _, _ = O.controller_step(O.controller_init(op), op, lr, h["mask"], h["so"], h["go"], seq, grp, batch,
                                       oadv)
    live = np.flatnonzero(host(coef) != 0)
    assert len(live) >= 4
    r_nan, r_inf, r_old, r_zero = (int(x) for x in live[:4])
    coef[r_zero] = 0.0
    ow[r_zero] = 0.0
    logits = b.logits.clone()
    logits[r_nan, 3] = float("nan")
    logits[r_inf, 5] = float("inf")
    logits[r_zero, :] = float("nan")
    old[r_old] = float("nan")
    z = rows_f64(logits, np.arange(b.T), b.V)
    olse, _, _, _ = O.token_stats(z, h["ids"], h["mask"])
    oold = host(old).astype(np.float64)
    coef_ref = O.loss_coefficients(ow, oadv, h["mask"], h["so"], seq, grp, batch, op)
    for recompute in (False, True):
        flags = api.new_flags()
        lse, _, _ = api.token_stats(logits, b.ids, b.mask, V=b.V)
        grad, tl, loss = api.loss_grad_logits(logits, b.ids, b.mask, None if recompute else lse, old, coef,
                                              p.clip_eps, V=b.V, flags=flags)
        assert api.read_flags(flags) & acrl.FLAG_NONFINITE
        ograd, otl, oloss = O.loss_grad_logits(z, h["ids"], h["mask"], None if recompute else olse, oold, oadv, ow,
                                               h["so"], seq, grp, batch, op)
        g = grad_rows(grad, np.arange(b.T), b.V)
        assert np.all(np.isnan(g[[r_nan, r_inf, r_old]])) and np.all(np.isnan(host(tl)[[r_nan, r_inf, r_old]]))
        assert np.all(g[r_zero] == 0.0) and float(host(tl)[r_zero]) == 0.0 and np.isnan(float(loss))
        assert_grad_rows(g, ograd, np.abs(coef_ref) * 2.0 + 1e-30, h["ids"], what=f"grad (recompute {recompute})")
        assert_close_rel(host(tl), otl, floor=1e-12, what="token_loss")


def test_chunked_gradient_matches_whole():
    spec = W.small_variant(W.GRPO, name="chunks", n_prompts=2, group_size=4, len_lo=30, len_hi=200, V=32000)
    b = _gen(spec, seed=4)
    p = acrl.Params()
    whole = acrl.AcrlStep.for_batch(b, p)
    whole.run_batch(b)
    chunked = acrl.AcrlStep.for_batch(b, p, grad_rows=100)
    got = torch.empty_like(whole.grad)

    def keep(r0, r1, g):
        got[r0:r1].copy_(g)
    chunked.run_batch(b, chunk_rows=100, on_chunk=keep)
    torch.cuda.synchronize()
    assert torch.equal(got[:, :b.V].view(torch.int16), whole.grad[:, :b.V].view(torch.int16))
    assert torch.equal(chunked.token_loss, whole.token_loss)
    assert float(chunked.loss) == float(whole.loss)


def test_bit_reproducible():
    spec = W.small_variant(W.QWEN, name="repro", n_prompts=2, group_size=3, len_lo=40, len_hi=90)
    b = _gen(spec, seed=8)
    outs = []
    for _ in range(2):
        s = acrl.AcrlStep.for_batch(b, acrl.Params())
        s.run_batch(b)
        torch.cuda.synchronize()
        outs.append((s.lse.clone(), s.entropy.clone(), s.weight.clone(), s.grad.clone(), s.loss.clone(),
                     s.disc.batch.clone()))
    for x, y in zip(*outs):
        assert torch.equal(x.view(torch.uint8) if x.dtype != torch.uint8 else x,
                           y.view(torch.uint8) if y.dtype != torch.uint8 else y)


# --------------------------------------------------------------------------
# edge cases and device flags
# --------------------------------------------------------------------------

def _tiny_manual(T, V, ld=None):
    ld = ld or ((V + 7) // 8) * 8
    gen = torch.Generator(device=DEV).manual_seed(T * 1000 + V)
    logits = torch.zeros((T, ld), dtype=torch.bfloat16, device=DEV)
    logits[:, :V] = (2 * torch.randn((T, V), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=gen, device=DEV, dtype=torch.int32)
    return logits, ids


@pytest.mark.parametrize("V", [1, 3, 7, 8, 9, 33, 16385])
def test_token_stats_odd_widths(V):
    T = 37
    logits, ids = _tiny_manual(T, V)
    lse, logp, H = api.token_stats(logits, ids, None, V=V)
    z = rows_f64(logits, np.arange(T), V)
    olse, ologp, oH, _ = O.token_stats(z, host(ids), None)
    assert_close_abs(host(logp), ologp, TOL_LOGP, "logp")
    assert_close_abs(host(lse), olse, TOL_LOGP, "lse")
    assert_close_rel(host(H), oH, floor=1e-5, what="H")


def test_empty_batch():
    logits = torch.zeros((0, 8), dtype=torch.bfloat16, device=DEV)
    ids = torch.zeros(0, dtype=torch.int32, device=DEV)
    lse, logp, H = api.token_stats(logits, ids, None, V=8)
    assert lse.numel() == 0


def test_bad_ids_nonfinite_and_masked_rows():
    T, V = 6, 40
    logits, ids = _tiny_manual(T, V)
    ids[1] = V          # out of range
    ids[2] = -1
    logits[3, 5] = float("nan")
    logits[4, 0] = float("-inf")
    mask = torch.ones(T, dtype=torch.uint8, device=DEV)
    mask[5] = 0
    logits[5, :] = float("nan")     # masked: never read
    flags = api.new_flags()
    lse, logp, H = api.token_stats(logits, ids, mask, V=V, flags=flags)
    f = api.read_flags(flags)
    assert f == (acrl.FLAG_BAD_ID | acrl.FLAG_NONFINITE)
    with pytest.raises(acrl.AcrlError, match="device flags raised: 0x3"):
        api.check_flags(flags)
    api.check_flags(api.new_flags())     # a clean word is ACRL_OK
    lp = host(logp)
    assert lp[1] == 0.0 and lp[2] == 0.0 and np.isnan(lp[3]) and np.isnan(host(H)[4]) and lp[5] == 0.0
    z = rows_f64(logits, np.arange(T), V)
    olse, ologp, oH, of = O.token_stats(z, host(ids), host(mask))
    assert of == f
    assert_close_abs(host(lse)[[0, 1, 2, 5]], olse[[0, 1, 2, 5]], TOL_LOGP, "lse")
    # the gradient kernel zeroes rows it cannot use and raises BAD_ID too
    coef = torch.full((T,), 0.01, device=DEV)
    flags2 = api.new_flags()
    grad, tl, loss = api.loss_grad_logits(logits, ids, mask, lse, None, coef, 0.2, V=V, flags=flags2)
    g = grad[:, :V].float()
    assert torch.all(g[1] == 0) and torch.all(g[2] == 0) and torch.all(g[5] == 0)
    assert api.read_flags(flags2) & acrl.FLAG_BAD_ID


def test_bad_offsets_flagged():
    T = 10
    lp = torch.zeros(T, device=DEV)
    so = torch.tensor([0, 6, 4, 10], dtype=torch.int64, device=DEV)
    go = torch.tensor([0, 3], dtype=torch.int32, device=DEV)
    flags = api.new_flags()
    api.seq_discrepancy(lp, lp, None, so, go, None, flags=flags)
    assert api.read_flags(flags) & acrl.FLAG_BAD_OFFSETS
    flags = api.new_flags()
    so = torch.tensor([0, 4, 9], dtype=torch.int64, device=DEV)      # does not reach T
    go = torch.tensor([0, 2], dtype=torch.int32, device=DEV)
    api.seq_discrepancy(lp, lp, None, so, go, None, flags=flags)
    assert api.read_flags(flags) & acrl.FLAG_BAD_OFFSETS
    flags = api.new_flags()
    so = torch.tensor([0, 4, 10], dtype=torch.int64, device=DEV)
    go = torch.tensor([0, 3], dtype=torch.int32, device=DEV)         # beyond S
    api.grpo_advantage(torch.zeros(2, device=DEV), go, acrl.Params(), flags=flags)
    assert api.read_flags(flags) & acrl.FLAG_BAD_OFFSETS


def test_invalid_arguments_rejected_on_host():
    logits, ids = _tiny_manual(4, 16)
    with pytest.raises(acrl.AcrlError):
        api.token_stats(logits[:, 1:], ids, None, V=15)        # misaligned rows
    with pytest.raises(acrl.AcrlError):
        api.grpo_advantage(torch.zeros(2, device=DEV), torch.tensor([0, 2], dtype=torch.int32, device=DEV),
                           acrl.Params(C=1.0))


# --------------------------------------------------------------------------
# controller trajectory: 50 steps with fresh batches (long-response shapes)
# --------------------------------------------------------------------------

def test_controller_trajectory_50_steps():
    spec = W.small_variant(W.LONG, name="traj", len_lo=512, len_hi=2048, perturb_frac=0.1, perturb_std=0.3)
    p = acrl.Params()
    op = oracle_params(p)
    state = api.controller_init(p)
    ost = O.controller_init(op)
    Xs = []
    for k in range(50):
        d = W.token_level(spec, W.seed_for("long", k), device=DEV)
        disc = api.seq_discrepancy(d["logp_pi"], d["logp_mu"], d["mask"], d["seq_offsets"], d["group_offsets"])
        adv = api.grpo_advantage(d["rewards"], d["group_offsets"], p)
        w, coef, alpha = api.controller_step(state, p, disc, d["mask"], d["seq_offsets"], d["group_offsets"], adv)
        torch.cuda.synchronize()
        lr, dd, seq, grp, batch, _ = O.seq_discrepancy(host(d["logp_pi"]).astype(np.float64),
                                                       host(d["logp_mu"]).astype(np.float64), host(d["mask"]),
                                                       host(d["seq_offsets"]), host(d["group_offsets"]))
        oadv = O.grpo_advantage(host(d["rewards"]).astype(np.float64), host(d["group_offsets"]), op)
        ow, oalpha, ost, info, _ = O.controller_step(ost, op, lr, host(d["mask"]), host(d["seq_offsets"]),
                                                     host(d["group_offsets"]), seq, grp, batch, oadv)
        st = api.read_state(state)
        assert int(st["step"]) == k + 1 and int(st["calibrated"]) == 1
        assert_close_rel(st["X"], ost.X, floor=1e-12, what=f"X step {k}")
        assert_close_rel(host(w), ow, floor=1e-7, what=f"weight step {k}")
        assert_close_rel(host(alpha), oalpha, floor=1e-6, what=f"alpha step {k}")
        Xs.append(float(st["X"]))
    assert all(x == Xs[0] for x in Xs)     # frozen after step 0, bit for bit


def test_cuda_graph_replay_matches_eager():
    """The step captured as a CUDA graph and replayed gives the eager step's outputs bit for bit."""
    spec = W.small_variant(W.GRPO, name="graph", n_prompts=2, group_size=4, len_lo=20, len_hi=200, V=32000)
    b = _gen(spec, seed=12)
    p = acrl.Params(X_init=0.013)     # a fixed X: every replay is the same computation
    eager = acrl.AcrlStep.for_batch(b, p)
    eager.run_batch(b)
    captured = acrl.AcrlStep.for_batch(b, p)
    graph = captured.capture(b)
    captured.grad.zero_()
    graph.replay()
    torch.cuda.synchronize()
    for x, y in ((eager.lse, captured.lse), (eager.weight, captured.weight), (eager.coef, captured.coef),
                 (eager.loss, captured.loss), (eager.grad, captured.grad)):
        assert torch.equal(x.view(torch.int16) if x.dtype == torch.bfloat16 else x,
                           y.view(torch.int16) if y.dtype == torch.bfloat16 else y)


def test_checkpoint_resume_is_bit_exact():
    """Save the controller state after 3 of 6 steps, restore it into a fresh state, and the last 3 steps'
    weights and states equal those of the uninterrupted run bit for bit."""
    spec = W.small_variant(W.LONG, name="ckpt", len_lo=64, len_hi=256, perturb_frac=0.2, perturb_std=0.3)
    p = acrl.Params(calib_steps=2, x_ema=0.25)

    def run(state, k0, k1):
        out = []
        for k in range(k0, k1):
            d = W.token_level(spec, W.seed_for("long", 100 + k), device=DEV)
            disc = api.seq_discrepancy(d["logp_pi"], d["logp_mu"], d["mask"], d["seq_offsets"], d["group_offsets"])
            adv = api.grpo_advantage(d["rewards"], d["group_offsets"], p)
            w, coef, alpha = api.controller_step(state, p, disc, d["mask"], d["seq_offsets"], d["group_offsets"], adv)
            out.append((w.clone(), api.save_state(state)))
        return out

    full = run(api.controller_init(p), 0, 6)
    s = api.controller_init(p)
    run(s, 0, 3)
    blob = api.save_state(s)
    resumed = run(api.load_state(blob), 3, 6)
    for (w1, s1), (w2, s2) in zip(full[3:], resumed):
        assert torch.equal(w1, w2) and s1 == s2


def test_bounded_wait_reports_timeout_and_context_survives():
    """A pipeline wait on a barrier nothing arrives on gives up after its limit and reports
    ACRL_FLAG_TIMEOUT; the context keeps working afterwards."""
    import time
    flags = api.new_flags()
    t0 = time.perf_counter()
    api.check(api.lib().acrl_selftest_wait_timeout(flags.data_ptr(), 50_000_000,
                                                   torch.cuda.current_stream().cuda_stream), "selftest")
    assert api.read_flags(flags) == acrl.FLAG_TIMEOUT
    assert time.perf_counter() - t0 < 30.0
    logits, ids = _tiny_manual(8, 64)
    lse, logp, H = api.token_stats(logits, ids, None, V=64)      # the context still runs kernels
    torch.cuda.synchronize()
    assert torch.all(torch.isfinite(lse))


def test_empty_batch_through_every_call():
    """T = 0, no responses, no prompts: every call accepts it and the outputs are zeros."""
    p = acrl.Params()
    step = acrl.AcrlStep(0, 64, 64, 0, 0, p)
    z = torch.zeros((0, 64), dtype=torch.bfloat16, device=DEV)
    e32 = torch.zeros(0, dtype=torch.int32, device=DEV)
    step.run(z, e32, torch.zeros(0, dtype=torch.uint8, device=DEV), torch.zeros(0, device=DEV),
             torch.zeros(0, device=DEV), torch.zeros(1, dtype=torch.int64, device=DEV),
             torch.zeros(1, dtype=torch.int32, device=DEV))
    torch.cuda.synchronize()
    b = step.batch_host()
    assert int(b["n_tokens"]) == 0 and int(b["n_groups_valid"]) == 0 and float(step.loss) == 0.0
    assert api.read_flags(step.flags) == acrl.FLAG_X_NONPOS     # nothing to calibrate X on


def test_fully_masked_batch():
    """Every token masked: zero statistics, weights, coefficients, gradient and loss; X cannot be calibrated."""
    spec = W.small_variant(W.GRPO, name="allmasked", n_prompts=2, group_size=3, len_lo=10, len_hi=40, V=3000)

    def mutate(b):
        b.mask.zero_()
    b = _gen(spec, seed=2, mutate=mutate)
    step = acrl.AcrlStep.for_batch(b, acrl.Params())
    step.grad.fill_(1.0)
    step.run_batch(b)
    torch.cuda.synchronize()
    assert torch.all(step.logp == 0) and torch.all(step.weight == 0) and torch.all(step.coef == 0)
    assert torch.all(step.grad[:, :b.V] == 0) and float(step.loss) == 0.0
    assert int(step.batch_host()["n_tokens"]) == 0
    assert api.read_flags(step.flags) == acrl.FLAG_X_NONPOS


def test_exchange_hook_as_two_identical_ranks():
    """The exchange hook sees the device bytes of the batch statistics between
    the discrepancy statistics and the controller.  An all-reduce over two
    ranks that hold the same batch doubles the three exchanged sums; doing
    that here must give the oracle's result on the batch concatenated with
    itself (one global X, the loss normalised by the global prompt count),
    restricted to the first copy."""
    from paper_2607_24062_gb300 import distributed as D
    spec = W.small_variant(W.GRPO, name="tworanks", n_prompts=3, group_size=4, len_lo=10, len_hi=120, V=3000,
                           perturb_frac=0.4, perturb_std=0.3)
    b = _gen(spec, seed=13)

    def as_two_ranks(buf):
        for name, dt in (("n_tokens", torch.int64), ("n_groups_valid", torch.int32), ("Y_sum", torch.float64)):
            D._field(buf, name, dt).mul_(2)

    params = acrl.Params()
    step = acrl.AcrlStep.for_batch(b, params)
    step.run_batch(b, exchange=as_two_ranks)
    torch.cuda.synchronize()
    h = _host_inputs(b)
    op = oracle_params(params)
    z = rows_f64(b.logits, np.arange(b.T), b.V)
    T, S = b.T, b.S
    cat = np.concatenate
    so2, go2 = cat([h["so"], h["so"][1:] + T]), cat([h["go"], h["go"][1:] + S]).astype(np.int32)
    ids2, mask2 = cat([h["ids"], h["ids"]]), cat([h["mask"], h["mask"]])
    res = O.step(cat([z, z]), ids2, mask2, cat([h["mu"], h["mu"]]), cat([h["R"], h["R"]]), so2, go2, op)
    gb = step.batch_host()
    assert int(gb["n_tokens"]) == res.batch["n_tokens"] and int(gb["n_groups_valid"]) == res.batch["n_groups_valid"]
    assert_close_rel(step.state_host()["X"], res.state.X, floor=1e-12, what="X")
    assert_close_rel(host(step.weight), res.weight[:T], floor=1e-7, what="weight")
    coef2 = O.loss_coefficients(res.weight, res.adv, mask2, so2, res.seq, res.grp, res.batch, op)
    assert_close_rel(host(step.coef), coef2[:T], floor=1e-12, what="coef")
    assert_close_rel(host(step.token_loss), res.token_loss[:T], floor=1e-12, what="token_loss")
    assert_loss(float(step.loss), 0.5 * res.loss, res.token_loss[:T])
    assert_grad_rows(grad_rows(step.grad, np.arange(T), b.V), res.grad[:T], coef2[:T], h["ids"])
    # without the exchange every coefficient would be twice as large
    assert np.any(np.abs(coef2[:T]) > 0)


def test_autograd_loss_through_an_lm_head():
    """acrl_loss as a torch.autograd node: loss.backward() delivers the
    kernel's dL/dlogits (bit for bit, and scaled by the incoming gradient),
    and it flows on into an upstream bf16 projection like any other grad."""
    spec = W.small_variant(W.GRPO, name="autograd", n_prompts=2, group_size=4, len_lo=20, len_hi=90, V=2048)
    b = _gen(spec, seed=21)
    step = acrl.AcrlStep.for_batch(b, acrl.Params())
    x = b.logits[:, :b.V].detach().requires_grad_(True)
    loss = acrl.acrl_loss(step, x, b.ids, b.mask, b.logp_mu, b.rewards, b.seq_offsets, b.group_offsets)
    loss.backward()
    torch.cuda.synchronize()
    assert torch.equal(x.grad.view(torch.int16), step.grad[:, :b.V].view(torch.int16))
    assert float(loss.detach()) == float(step.loss)
    x.grad = None
    (2.0 * acrl.acrl_loss(step, x, b.ids, b.mask, b.logp_mu, b.rewards, b.seq_offsets, b.group_offsets)).backward()
    assert torch.equal(x.grad.float(), 2.0 * step.grad[:, :b.V].float())
    # an LM head upstream: logits = h W^T in bf16; W's gradient is g^T h
    K = 64
    gen = torch.Generator(device=DEV).manual_seed(5)
    h = torch.randn((b.T, K), generator=gen, device=DEV).to(torch.bfloat16)
    Wt = (0.1 * torch.randn((b.V, K), generator=gen, device=DEV)).to(torch.bfloat16).requires_grad_(True)
    logits = h @ Wt.t()
    step2 = acrl.AcrlStep(b.T, b.V, b.V, b.S, b.Gn, acrl.Params())
    acrl.acrl_loss(step2, logits, b.ids, b.mask, b.logp_mu, b.rewards, b.seq_offsets, b.group_offsets).backward()
    ref = step2.grad.float().t() @ h.float()
    assert torch.allclose(Wt.grad.float(), ref, rtol=2e-2, atol=1e-6 + 2e-2 * float(ref.abs().max()))


def _quadrant_rows():
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "acrl_quadrants.txt")
    with open(path) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


def _one_token_controller(pi, mu, A, X, **kw):
    """One prompt with one response of one token, fed to the O(T) calls as
    log-probs: Y = D = |pi - mu|, A = R (a singleton prompt), X given."""
    p = acrl.Params(X_init=X, **kw)
    f32 = dict(dtype=torch.float32, device=DEV)
    so = torch.tensor([0, 1], dtype=torch.int64, device=DEV)
    go = torch.tensor([0, 1], dtype=torch.int32, device=DEV)
    disc = api.seq_discrepancy(torch.tensor([math.log(pi)], **f32), torch.tensor([math.log(mu)], **f32), None, so, go)
    adv = api.grpo_advantage(torch.tensor([A], **f32), go, p)
    w, coef, alpha = api.controller_step(api.controller_init(p), p, disc, None, so, go, adv)
    return float(w[0]), float(alpha[0]), float(disc.grp_host()[0]["Y"]), p


@pytest.mark.parametrize("row", _quadrant_rows(), ids=lambda r: f"{r[0]}-{r[1]}")
def test_sign_table_on_gpu(row):
    """Sec. 4.2's eight cases on the GPU: the sign of alpha and whether the
    weight is above or below 1, for Y > X and Y < X in each (A, pi vs mu)."""
    regime, _, sA, pvm, salpha, rho_vs = row[:6]
    pi, mu = (0.3, 0.5) if pvm == "<" else (0.5, 0.3)
    X = 0.1 if regime == "Y>X" else 0.4                      # Y = |pi - mu| = 0.2
    w, alpha, Y, p = _one_token_controller(pi, mu, 1.0 if sA == "+" else -1.0, X)
    assert Y == pytest.approx(0.2, rel=1e-6)
    assert alpha != 0.0 and (alpha > 0) == (salpha == "+")
    assert (w > 1.0) == (rho_vs == ">")
    assert w == pytest.approx(min((pi / mu) ** alpha, p.C), rel=2e-6)


def test_controller_special_cases_on_gpu():
    # Y = X: X set to the Y the GPU computed, so alpha is exactly 0 and the weight exactly 1
    _, _, Y, _ = _one_token_controller(0.2, 0.4, 1.0, 1.0)
    w, alpha, _, _ = _one_token_controller(0.2, 0.4, 1.0, Y)
    assert alpha == 0.0 and w == 1.0
    w, alpha, _, _ = _one_token_controller(0.2, 0.4, 0.0, 0.013)     # A = 0
    assert alpha == 0.0 and w == 1.0
    w, alpha, _, _ = _one_token_controller(0.3, 0.3, 1.0, 0.013)     # mu = pi: rho = 1 for any alpha
    assert w == 1.0


def test_calibration_over_prompts_of_two_batches_on_gpu():
    """calib_steps = 2 over batches of 1 and 3 prompts: X is the mean of Y_g
    over all four prompts (Sec. 4.1), not the mean of the two batch means."""
    p = acrl.Params(calib_steps=2)
    op = oracle_params(p)
    state, ost = api.controller_init(p), O.controller_init(op)
    f32 = dict(dtype=torch.float32, device=DEV)
    Ys = []
    for G, mu in ((1, 0.31), (3, 0.36)):
        lp_pi = torch.full((G,), math.log(0.3), **f32)
        lp_mu = torch.full((G,), math.log(mu), **f32)
        so = torch.arange(G + 1, dtype=torch.int64, device=DEV)
        go = torch.arange(G + 1, dtype=torch.int32, device=DEV)
        disc = api.seq_discrepancy(lp_pi, lp_mu, None, so, go)
        adv = api.grpo_advantage(torch.ones(G, **f32), go, p)
        api.controller_step(state, p, disc, None, so, go, adv)
        lr, d, seq, grp, batch, _ = O.seq_discrepancy(host(lp_pi).astype(np.float64), host(lp_mu).astype(np.float64),
                                                      None, host(so), host(go))
        ost = O.controller_step(ost, op, lr, None, host(so), host(go), seq, grp, batch, np.ones(G))[2]
        Ys.append(list(disc.grp_host()["Y"]))
    st = api.read_state(state)
    assert bool(st["calibrated"]) and ost.calibrated
    assert_close_rel(float(st["X"]), ost.X, floor=1e-12, what="X")
    by_prompt = (sum(Ys[0]) + sum(Ys[1])) / 4
    assert float(st["X"]) == pytest.approx(by_prompt, rel=1e-12)
    assert abs(by_prompt - (np.mean(Ys[0]) + np.mean(Ys[1])) / 2) > 1e-3 * by_prompt


def test_infinite_and_nan_rollout_log_probs_on_gpu():
    """mu = 0 on a sampled token (log mu = -inf) and a NaN log-prob, fed to
    the O(T) calls: the weights and flags the oracle gives."""
    f32 = dict(dtype=torch.float32, device=DEV)
    so = torch.tensor([0, 1, 2, 3], dtype=torch.int64, device=DEV)
    go = torch.tensor([0, 1, 2, 3], dtype=torch.int32, device=DEV)
    lp_pi = torch.tensor([-1.0, -1.0, -1.0], **f32)
    lp_mu = torch.tensor([-math.inf, -math.inf, math.nan], **f32)
    for mode, A in ((acrl.MODE_ACRL, (0.0, 1.0, -1.0)), (acrl.MODE_TIS, (1.0, 1.0, 1.0)),
                    (acrl.MODE_MIS, (1.0, -1.0, 1.0))):
        p = acrl.Params(mode=mode, X_init=0.1)
        op = oracle_params(p)
        flags = api.new_flags()
        disc = api.seq_discrepancy(lp_pi, lp_mu, None, so, go, flags=flags)
        adv = torch.tensor(A, **f32)
        w, coef, alpha = api.controller_step(api.controller_init(p), p, disc, None, so, go, adv, flags=flags)
        lr, d, seq, grp, batch, of = O.seq_discrepancy(host(lp_pi).astype(np.float64), host(lp_mu).astype(np.float64),
                                                       None, host(so), host(go))
        ow, oalpha, *_ = O.controller_step(O.controller_init(op), op, lr, None, host(so), host(go), seq, grp, batch,
                                           np.array(A))
        assert api.read_flags(flags) & acrl.FLAG_NONFINITE and of & O.FLAG_NONFINITE
        np.testing.assert_allclose(host(w), ow, rtol=1e-6, atol=0, err_msg=f"mode {mode}")
        assert host(w)[2] == 0.0


@pytest.mark.parametrize("mode", [acrl.MODE_ACRL, acrl.MODE_MIS])
def test_importance_weights_from_log_probs(mode):
    """The weights-only call (log-probs in, weights out) against the oracle's
    discrepancy, advantage and controller stages, over three batches (the
    first calibrates X)."""
    spec = W.small_variant(W.GRPO, name="weights_only", n_prompts=4, group_size=4, len_lo=5, len_hi=90,
                           perturb_frac=0.3, perturb_std=0.3)
    p = acrl.Params(mode=mode)
    op = oracle_params(p)
    state, ostate = api.controller_init(p), O.controller_init(op)
    for k in range(3):
        d = W.token_level(spec, 700 + k, device=DEV)
        r = acrl.importance_weights(state, p, d["logp_pi"], d["logp_mu"], d["mask"], d["rewards"], d["seq_offsets"],
                                    d["group_offsets"])
        mask, so, go = host(d["mask"]), host(d["seq_offsets"]), host(d["group_offsets"])
        lr, dd, seq, grp, batch, f = O.seq_discrepancy(host(d["logp_pi"]).astype(np.float64),
                                                        host(d["logp_mu"]).astype(np.float64), mask, so, go)
        adv = O.grpo_advantage(host(d["rewards"]).astype(np.float64), go, op)
        w, alpha, ostate, info, f2 = O.controller_step(ostate, op, lr, mask, so, go, seq, grp, batch, adv)
        assert api.read_flags(r.flags) == (f | f2)
        compare_seq(r.disc.seq_host(), seq)
        assert_close_rel(host(r.adv), adv, floor=1e-6, what="adv")
        assert_close_rel(host(r.alpha), alpha, floor=1e-6, what="alpha")
        assert_close_rel(host(r.weight), w, floor=1e-7, what="weight")
        coef = O.loss_coefficients(w, adv, mask, so, seq, grp, batch, op)
        assert_close_rel(host(r.coef), coef, floor=1e-12, what="coef")
        assert_close_rel(api.read_state(state)["X"], ostate.X, floor=1e-12, what="X")


@pytest.mark.parametrize("V", [1, 7, 8, 9, 4096, 4097, 6144, 6151, 6152, 16383, 16384, 16385, 20480, 24576, 24583, 24584,
                               32000, 36864, 36871, 36872, 40960, 40967, 40968, 49152, 49153, 49160, 65535, 65536,
                               65537, 65544, 81920, 100000, 114688, 114695])
def test_row_size_class_boundaries(V):
    """Vocabularies at the edges of the row-team size classes (eight lanes up
    to 4,096 columns, one warp up to 16,384, 64 threads up to 65,536, 128
    above for the statistics;
    one warp, then 512 threads, then 768 above 65,536 for the gradient; one
    warp up to 6,144 columns, 128 threads up to 24,583, 256 up to 40,967,
    then 512 for the gradient with the lse recomputed), of the 8-column
    vectors and of the parts of a row the recompute path holds on chip
    (20,480 columns in shared memory for 128-thread CTAs, 36,864 for 256-
    thread ones, 49,152 for 512-thread ones, then whole chunks of 16,384
    columns in tensor memory: 0 to 4 chunks, with and without a ragged tail):
    statistics and gradient against the oracle on every element, with the lse
    recomputed in the gradient kernel as well."""
    T = 37
    ld = ((V + 7) // 8) * 8
    gen = torch.Generator(device=DEV).manual_seed(V)
    logits = (2.0 * torch.randn((T, ld), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, V, (T,), generator=gen, device=DEV, dtype=torch.int32)
    mask = (torch.rand(T, generator=gen, device=DEV) < 0.85).to(torch.uint8)
    coef = torch.randn(T, generator=gen, device=DEV) * mask.float()
    flags = api.new_flags()
    lse, logp, H = api.token_stats(logits, ids, mask, V=V, flags=flags)
    z = rows_f64(logits, np.arange(T), V)
    olse, ologp, oH, _ = O.token_stats(z, host(ids), host(mask))
    assert_close_abs(host(lse), olse, TOL_LOGP, "lse")
    assert_close_abs(host(logp), ologp, TOL_LOGP, "logp")
    assert_close_rel(host(H), oH, floor=1e-5, what="entropy")
    m = host(mask).astype(bool)
    p = np.exp(z - olse[:, None])
    onehot = np.zeros((T, V))
    onehot[np.arange(T), host(ids)] = 1.0
    want = host(coef).astype(np.float64)[:, None] * (p - onehot)
    want[~m] = 0.0
    for recompute in (False, True):
        grad, _, _ = api.loss_grad_logits(logits, ids, mask, None if recompute else lse, None, coef, 0.2, V=V,
                                          flags=flags)
        assert_grad_rows(grad_rows(grad, np.arange(T), V), want, host(coef), host(ids), what=f"grad (recompute "
                         f"{recompute})")
    assert api.read_flags(flags) == 0


@pytest.mark.parametrize("offset", [0, 1])
def test_loss_sum_blocks_tails_and_alignment(offset):
    """acrl_reduce_loss (the scalar loss of Eq. ACRL's sum over tokens):
    lengths at the edges of the eight CTAs' blocks of float4 groups and of the
    ragged tail, from a 16-byte-aligned array and from one starting an element
    later (the scalar path): the fp32 result agrees with math.fsum of the same
    values within the rounding of fp32 groups of four, and two calls agree
    bit for bit."""
    gen = torch.Generator(device=DEV).manual_seed(5 + offset)
    base = torch.randn(600_000, generator=gen, device=DEV)
    for T in (0, 1, 3, 4, 5, 31, 32, 33, 1023, 1024, 1025, 32767, 32768, 32769, 147831, 524288 + 7):
        x = base[offset: offset + T]
        a = api.reduce_loss(x)
        b = api.reduce_loss(x)
        torch.cuda.synchronize()
        assert torch.equal(a, b), T
        ref = math.fsum(host(x).astype(np.float64).tolist())
        bound = 1e-6 * float(host(x).astype(np.float64).__abs__().sum()) + 1e-6
        assert abs(float(a) - ref) <= bound, (T, float(a), ref)
