"""The pins must catch plausible mistakes in the oracle.  Each case plants one
mistake in a copy of an oracle function (on the CPU) and runs the pins of
that function: at least one of them must fail.  Nothing here touches the GPU
path."""

import numpy as np
import pytest

import oracle as O
import oracle.acrl_oracle as OA
import test_oracle_pins as P


def _token_stats_entropy_sign(z, ids, mask):
    lse, logp, H, f = OA._orig["token_stats"](z, ids, mask)
    return lse, logp, -H, f


def _token_stats_logp_index(z, ids, mask):
    lse, logp, H, f = OA._orig["token_stats"](z, np.clip(np.asarray(ids) + 1, 0, np.asarray(z).shape[1] - 1), mask)
    return lse, logp, H, f


def _recompute_d_log(logp_pi, logp_mu, mask, so, go, entropy=None):
    """Mistake: d taken on log-probabilities, |log pi - log mu|, instead of probabilities."""
    lr, d, seq, grp, batch, f = OA._orig["seq_discrepancy"](logp_pi, logp_mu, mask, so, go, entropy)
    d2 = np.abs(np.asarray(logp_pi, dtype=float) - np.asarray(logp_mu, dtype=float))
    m = np.ones(len(d2), dtype=bool) if mask is None else np.asarray(mask) != 0
    d2 = np.where(m, d2, 0.0)
    so = np.asarray(so)
    for i in range(len(so) - 1):
        sl = slice(so[i], so[i + 1])
        if seq["n"][i]:
            seq["mean_d"][i] = d2[sl][m[sl]].sum() / seq["n"][i]
    for g in range(len(go) - 1):
        members = [i for i in range(go[g], go[g + 1]) if seq["n"][i] > 0]
        grp["Y"][g] = sum(seq["mean_d"][i] for i in members) / len(members) if members else 0.0
    return lr, d2, seq, grp, batch, f


def _grpo_ddof_ignored(rewards, group_offsets, params):
    p = O.Params(**{**vars(params), "adv_ddof": 0})
    return OA._orig["grpo_advantage"](rewards, group_offsets, p)


def _grpo_no_centering(rewards, group_offsets, params):
    A = OA._orig["grpo_advantage"](rewards, group_offsets, params)
    return A + 0.1


def _controller_alpha_sign(state, params, *args):
    p = O.Params(**{**vars(params), "gamma": -params.gamma})
    return OA._orig["controller_step"](state, p, *args)


def _controller_no_truncation(state, params, *args):
    p = O.Params(**{**vars(params), "C": 1e30})
    return OA._orig["controller_step"](state, p, *args)


def _loss_grad_sign(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params, rows=None):
    """Mistake: gradient of J instead of L = -J (sign flipped)."""
    grad, tl, loss = OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp,
                                                  batch, params, rows)
    return -grad, tl, loss


def _loss_grad_wrong_column(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params,
                            rows=None):
    """Mistake: the one-hot subtracted at the neighbouring column."""
    V = np.asarray(z).shape[1]
    shifted = (np.asarray(ids) + 1) % V
    grad, tl, loss = OA._orig["loss_grad_logits"](z, shifted, mask, lse, old_logp, adv, weight, seq_offsets, seq,
                                                  grp, batch, params, rows)
    return grad, tl, loss


def _loss_grad_no_norm(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params, rows=None):
    b2 = dict(batch)
    b2["n_groups_valid"] = 1
    return OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, b2, params,
                                        rows)


def _controller_continuous_sign(state, params, *args):
    """Mistake: the continuous-reduction ablation raises the weight it should lower."""
    if params.mode == O.MODE_ACRL_CONTINUOUS:
        params = O.Params(**{**vars(params), "kappa": -params.kappa})
    return OA._orig["controller_step"](state, params, *args)


def _controller_no_moving_average(state, params, *args):
    """Mistake: the moving-average X never moves."""
    return OA._orig["controller_step"](state, O.Params(**{**vars(params), "x_ema": 0.0}), *args)


def _controller_calibration_by_batch(state, params, lr, mask, so, go, seq, grp, batch, adv):
    """Mistake: X as the mean of the calibration batches' means instead of over all their prompts."""
    b2 = dict(batch)
    b2["Y_sum"] = batch["Y_mean"]
    b2["n_groups_valid"] = 1 if batch["n_groups_valid"] > 0 else 0
    return OA._orig["controller_step"](state, params, lr, mask, so, go, seq, grp, b2, adv)


def _loss_grad_entropy_sign(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params, rows=None):
    """Mistake: the entropy bonus penalises entropy."""
    p = O.Params(**{**vars(params), "entropy_coeff": -params.entropy_coeff})
    return OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, p,
                                        rows)


def _discrepancy_token_weighted_Y(logp_pi, logp_mu, mask, so, go, entropy=None):
    """Mistake: Y_g as the token mean of d over the prompt instead of the mean of its responses' D_i."""
    lr, d, seq, grp, batch, f = OA._orig["seq_discrepancy"](logp_pi, logp_mu, mask, so, go, entropy)
    for g in range(len(go) - 1):
        members = [i for i in range(go[g], go[g + 1]) if seq["n"][i] > 0]
        ntok = sum(seq["n"][i] for i in members)
        grp["Y"][g] = sum(seq["mean_d"][i] * seq["n"][i] for i in members) / ntok if ntok else 0.0
    return lr, d, seq, grp, batch, f


def _lmhead_not_rounded(hidden, weight):
    """Mistake: the logits kept at full precision instead of the engine's bf16."""
    return np.asarray(hidden, dtype=np.float64) @ np.asarray(weight, dtype=np.float64).T


def _round_bf16_truncates(x):
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    return np.ldexp(np.trunc(f * 256.0) / 256.0, e)


def _grpo_singleton_zero(rewards, group_offsets, params):
    """Mistake: a prompt with one response gets A = 0 under the mean-0/std-1 rule."""
    p = O.Params(**{**vars(params), "singleton_rule": O.SINGLETON_ZERO})
    return OA._orig["grpo_advantage"](rewards, group_offsets, p)


def _controller_zero_alpha_unguarded(state, params, lr, mask, so, go, seq, grp, batch, adv):
    """Mistake: rho^alpha evaluated as exp(alpha * lr) with no alpha = 0 case, so that
    alpha = 0 on a token with lr = +inf gives exp(0 * inf) = NaN instead of 1."""
    w, alpha, st, info, f = OA._orig["controller_step"](state, params, lr, mask, so, go, seq, grp, batch, adv)
    w = np.array(w, dtype=np.float64)
    lr = np.asarray(lr, dtype=np.float64)
    for i in range(len(so) - 1):
        for t in range(int(so[i]), int(so[i + 1])):
            valid = mask is None or mask[t] != 0
            if valid and params.mode != O.MODE_MIS and alpha[i] == 0.0 and np.isinf(lr[t]):
                w[t] = np.nan
    return w, alpha, st, info, f


def _controller_nan_weight_one(state, params, lr, mask, so, go, seq, grp, batch, adv):
    """Mistake: a token whose log-ratio is NaN keeps weight 1 instead of 0."""
    w, alpha, st, info, f = OA._orig["controller_step"](state, params, lr, mask, so, go, seq, grp, batch, adv)
    w = np.array(w, dtype=np.float64)
    lr = np.asarray(lr, dtype=np.float64)
    nan = np.isnan(lr) if mask is None else np.isnan(lr) & (np.asarray(mask) != 0)
    w[nan] = 1.0
    return w, alpha, st, info, f


def _loss_grad_no_clip(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params, rows=None):
    """Mistake: the PPO clip left out (min(r A, clip(r) A) taken as r A everywhere)."""
    p = O.Params(**{**vars(params), "clip_eps": 1e9})
    return OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, p,
                                        rows)


def _controller_y_per_response(state, params, *args):
    """Mistake: Y read per response (D_i) where the prompt mean Y_g is the default."""
    if params.y_gran == O.Y_GROUP:
        params = O.Params(**{**vars(params), "y_gran": O.Y_SEQUENCE})
    return OA._orig["controller_step"](state, params, *args)


def _controller_mis_mean_ratio(state, params, lr, mask, so, go, seq, grp, batch, adv):
    """Mistake: the sequence ratio of MIS from the mean token log-ratio instead of the sum."""
    seq2 = dict(seq)
    n = np.maximum(np.asarray(seq["n"]), 1)
    seq2["sum_lr"] = np.asarray(seq["sum_lr"], dtype=np.float64) / n
    return OA._orig["controller_step"](state, params, lr, mask, so, go, seq2, grp, batch, adv)


def _token_stats_lse_without_max(z, ids, mask):
    """Mistake: the row maximum subtracted for stability never added back."""
    lse, logp, H, f = OA._orig["token_stats"](z, ids, mask)
    mx = np.asarray(z, dtype=np.float64).max(axis=1)
    m = np.ones(len(lse), dtype=bool) if mask is None else np.asarray(mask) != 0
    return np.where(m, lse - mx, lse), np.where(m, logp + mx, logp), np.where(m, H - mx, H), f


def _regroup(seq, grp, go, divisor):
    for g in range(len(go) - 1):
        members = list(range(go[g], go[g + 1]))
        valid = [i for i in members if seq["n"][i] > 0]
        den = divisor(members, valid)
        grp["Y"][g] = sum(seq["mean_d"][i] for i in valid) / den if den else 0.0


def _discrepancy_mean_over_all_rows(logp_pi, logp_mu, mask, so, go, entropy=None):
    """Mistake: D_i divides by every row of the response, masked padding included."""
    lr, d, seq, grp, batch, f = OA._orig["seq_discrepancy"](logp_pi, logp_mu, mask, so, go, entropy)
    so = np.asarray(so)
    for i in range(len(so) - 1):
        if seq["n"][i] > 0:
            seq["mean_d"][i] = seq["sum_d"][i] / (so[i + 1] - so[i])
    _regroup(seq, grp, go, lambda members, valid: len(valid))
    return lr, d, seq, grp, batch, f


def _discrepancy_empty_responses_counted(logp_pi, logp_mu, mask, so, go, entropy=None):
    """Mistake: G_g counts the responses with no valid token."""
    lr, d, seq, grp, batch, f = OA._orig["seq_discrepancy"](logp_pi, logp_mu, mask, so, go, entropy)
    _regroup(seq, grp, go, lambda members, valid: len(members) if valid else 0)
    return lr, d, seq, grp, batch, f


def _grpo_no_eps(rewards, group_offsets, params):
    """Mistake: adv_eps left out of the denominator."""
    return OA._orig["grpo_advantage"](rewards, group_offsets, O.Params(**{**vars(params), "adv_eps": 0.0}))


def _controller_never_frozen(state, params, *args):
    """Mistake: X recalibrated on every batch instead of frozen after calibration."""
    if params.X_init <= 0 and state.calibrated:
        state.calibrated = False
        state.calib_sum, state.calib_count, state.calib_done_steps = 0.0, 0, 0
    return OA._orig["controller_step"](state, params, *args)


def _loss_grad_token_mean(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params, rows=None):
    """Mistake: the default sequence-mean-token-mean aggregation replaced by a token mean."""
    if params.agg == O.AGG_SEQ_MEAN_TOKEN_MEAN:
        params = O.Params(**{**vars(params), "agg": O.AGG_TOKEN_MEAN})
    return OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch,
                                        params, rows)


def _round_bf16_half_away(x):
    """Mistake: ties rounded away from zero instead of to even."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    return np.ldexp(np.trunc(f * 256.0 + np.copysign(0.5, f)) / 256.0, e)


def _token_stats_no_bad_id_flag(z, ids, mask):
    """Mistake: an id outside [0, V) is not reported."""
    lse, logp, H, f = OA._orig["token_stats"](z, ids, mask)
    return lse, logp, H, f & ~O.FLAG_BAD_ID


def _discrepancy_no_offsets_flag(logp_pi, logp_mu, mask, so, go, entropy=None):
    """Mistake: inconsistent offsets are not reported."""
    lr, d, seq, grp, batch, f = OA._orig["seq_discrepancy"](logp_pi, logp_mu, mask, so, go, entropy)
    return lr, d, seq, grp, batch, f & ~O.FLAG_BAD_OFFSETS


def _controller_no_x_flag(state, params, *args):
    """Mistake: X <= 0 is not reported."""
    w, alpha, st, info, f = OA._orig["controller_step"](state, params, *args)
    return w, alpha, st, info, f & ~O.FLAG_X_NONPOS


PIN_GROUPS = {
    "token_stats": [lambda: P.test_token_stats_matches_bruteforce(7), P.test_token_stats_library_routines,
                    P.test_two_way_closed_form, P.test_mask_nonfinite_and_bad_id],
    "seq_discrepancy": [P.test_distance_is_on_probabilities, P.test_hand_worked_aggregates,
                        P.test_aggregates_as_linear_functional, P.test_bad_offsets_flagged],
    "grpo_advantage": [lambda: P.test_grpo_binary_closed_form(8, 3), P.test_grpo_matches_scipy_zscore,
                       P.test_grpo_special_groups],
    "controller_step": [lambda: [P.test_quadrant_sign_table(r) for r in P._read_quadrants()],
                        P.test_controller_special_cases, P.test_tis_and_mis_thresholds,
                        lambda: [P.test_continuous_reduction_always_reduces(r) for r in P._read_quadrants()],
                        P.test_continuous_reduction_kappa, P.test_moving_average_X_by_hand,
                        P.test_calibration_averages_prompts_across_batches, P.test_infinite_and_nan_log_ratios,
                        P.test_y_granularity_options, P.test_mis_sequence_ratio_is_product,
                        P.test_calibration_then_frozen, P.test_nonpositive_X_flag_and_fixed_point],
    "loss_grad_logits": [lambda: P.test_gradient_matches_autograd(False, 0.0), P.test_on_policy_loss_by_hand_and_invariants,
                         lambda: P.test_gradient_central_differences(0.0), P.test_entropy_bonus_by_hand,
                         lambda: P.test_gradient_matches_autograd(True, 0.0), P.test_clip_gate,
                         lambda: P.test_gradient_undefined_rows(True), lambda: P.test_gradient_undefined_rows(False)],
    "round_bf16": [P.test_round_bf16_matches_library_and_ties],
    "lmhead_logits": [P.test_lmhead_logits_small],
}

def _loss_grad_undefined_rows_zero(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch, params,
                                   rows=None):
    """Mistake: a row the call cannot evaluate gets a zero gradient row and token loss 0 instead of NaN."""
    grad, tl, loss = OA._orig["loss_grad_logits"](z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp,
                                                  batch, params, rows=rows)
    bad = np.isnan(tl)
    tl = np.where(bad, 0.0, tl)
    return np.where(np.isnan(grad), 0.0, grad), tl, float(np.sum(tl[~np.isnan(tl)]))


MUTATIONS = [
    ("token_stats", "entropy sign flipped", _token_stats_entropy_sign),
    ("token_stats", "log-prob of the wrong column", _token_stats_logp_index),
    ("seq_discrepancy", "distance on log-probabilities", _recompute_d_log),
    ("grpo_advantage", "std with ddof 0 instead of 1", _grpo_ddof_ignored),
    ("grpo_advantage", "advantage not centred", _grpo_no_centering),
    ("controller_step", "alpha with the wrong sign", _controller_alpha_sign),
    ("controller_step", "weights never truncated at C", _controller_no_truncation),
    ("loss_grad_logits", "gradient sign flipped", _loss_grad_sign),
    ("loss_grad_logits", "one-hot at the wrong column", _loss_grad_wrong_column),
    ("loss_grad_logits", "prompt count left out of the normalisation", _loss_grad_no_norm),
    ("round_bf16", "truncation instead of round-to-nearest-even", _round_bf16_truncates),
    ("controller_step", "continuous reduction with the opposite sign", _controller_continuous_sign),
    ("controller_step", "moving-average X never applied", _controller_no_moving_average),
    ("controller_step", "X from the mean of batch means", _controller_calibration_by_batch),
    ("loss_grad_logits", "entropy bonus with the wrong sign", _loss_grad_entropy_sign),
    ("seq_discrepancy", "Y_g weighted by tokens instead of responses", _discrepancy_token_weighted_Y),
    ("lmhead_logits", "logits not rounded to bf16", _lmhead_not_rounded),
    ("grpo_advantage", "lone response given no advantage", _grpo_singleton_zero),
    ("controller_step", "alpha = 0 with an infinite log-ratio gives NaN", _controller_zero_alpha_unguarded),
    ("controller_step", "NaN log-ratio keeps weight 1", _controller_nan_weight_one),
    ("loss_grad_logits", "PPO clip left out", _loss_grad_no_clip),
    ("controller_step", "Y per response instead of per prompt", _controller_y_per_response),
    ("controller_step", "MIS ratio from the mean log-ratio", _controller_mis_mean_ratio),
    ("token_stats", "row maximum never added back to lse", _token_stats_lse_without_max),
    ("seq_discrepancy", "D_i over every row, padding included", _discrepancy_mean_over_all_rows),
    ("seq_discrepancy", "empty responses counted in G_g", _discrepancy_empty_responses_counted),
    ("grpo_advantage", "adv_eps left out", _grpo_no_eps),
    ("controller_step", "X recalibrated every batch", _controller_never_frozen),
    ("loss_grad_logits", "token mean instead of sequence mean", _loss_grad_token_mean),
    ("round_bf16", "ties away from zero", _round_bf16_half_away),
    ("token_stats", "bad id not reported", _token_stats_no_bad_id_flag),
    ("seq_discrepancy", "bad offsets not reported", _discrepancy_no_offsets_flag),
    ("controller_step", "X <= 0 not reported", _controller_no_x_flag),
    ("loss_grad_logits", "undefined rows given a zero gradient", _loss_grad_undefined_rows_zero),
]


@pytest.fixture
def mutate(monkeypatch):
    if not hasattr(OA, "_orig"):
        OA._orig = {name: getattr(OA, name) for name in PIN_GROUPS}

    def apply(name, fn):
        monkeypatch.setattr(OA, name, fn)
        monkeypatch.setattr(O, name, fn)
        monkeypatch.setattr(P.O, name, fn)
    return apply


@pytest.mark.parametrize("target,what,fn", MUTATIONS, ids=[m[1] for m in MUTATIONS])
def test_pins_catch_planted_mistake(mutate, target, what, fn):
    mutate(target, fn)
    caught = 0
    for pin in PIN_GROUPS[target]:
        try:
            pin()
        except AssertionError:
            caught += 1
    assert caught > 0, f"no pin caught: {what}"


def test_unmutated_oracle_passes_the_same_pins():
    for pins in PIN_GROUPS.values():
        for pin in pins:
            pin()
