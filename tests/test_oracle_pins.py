"""Pins for the float64 oracle: each test checks it against something other
than its own formulas -- brute force with math.fsum, closed forms, library
routines (scipy, torch autograd), invariants, hand-worked numbers and the sign
table printed in Sec. 4.2 of the paper.  CPU only."""

import math
import os

import numpy as np
import pytest
import scipy.special
import scipy.stats
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# a1 token statistics
# --------------------------------------------------------------------------

@pytest.mark.parametrize("V", [2, 7, 64])
def test_token_stats_matches_bruteforce(V):
    rng = np.random.default_rng(V)
    T = 24
    z = rng.normal(0, 3, size=(T, V))
    ids = rng.integers(0, V, size=T)
    lse, logp, H, flags = O.token_stats(z, ids, None)
    blse, blogp, bH = O.token_stats_bruteforce(z, ids)
    assert flags == 0
    np.testing.assert_allclose(lse, blse, rtol=0, atol=1e-12)
    np.testing.assert_allclose(logp, blogp, rtol=0, atol=1e-12)
    np.testing.assert_allclose(H, bH, rtol=0, atol=1e-12)


def test_token_stats_library_routines():
    rng = np.random.default_rng(1)
    z = rng.standard_t(4, size=(16, 301)) * 2
    ids = rng.integers(0, 301, size=16)
    lse, logp, H, _ = O.token_stats(z, ids, None)
    np.testing.assert_allclose(lse, scipy.special.logsumexp(z, axis=1), atol=1e-12)
    p = scipy.special.softmax(z, axis=1)
    np.testing.assert_allclose(H, scipy.stats.entropy(p, axis=1), atol=1e-10)
    np.testing.assert_allclose(logp, np.log(p[np.arange(16), ids]), atol=1e-12)


@pytest.mark.parametrize("V", [1, 2, 4096, 151936])
def test_uniform_logits(V):
    z = np.full((2, V), 0.37)
    lse, logp, H, _ = O.token_stats(z, np.array([0, V - 1]), None)
    np.testing.assert_allclose(logp, -math.log(V), atol=1e-12)
    np.testing.assert_allclose(H, math.log(V), atol=1e-9)
    np.testing.assert_allclose(lse, 0.37 + math.log(V), atol=1e-12)


def test_one_hot_dominant_and_shift():
    V = 50
    z = np.zeros((2, V))
    z[0, 7] = 1000.0
    z[1] = np.linspace(-3, 5, V)
    lse, logp, H, _ = O.token_stats(z, np.array([7, 3]), None)
    assert abs(logp[0]) < 1e-300 or logp[0] == 0.0
    assert H[0] < 1e-300 * 1e10 or H[0] == 0.0
    lse2, logp2, H2, _ = O.token_stats(z + 123.25, np.array([7, 3]), None)
    np.testing.assert_allclose(logp2, logp, atol=1e-12)
    np.testing.assert_allclose(H2, H, atol=1e-12)
    np.testing.assert_allclose(lse2, lse + 123.25, atol=1e-12)


def test_two_way_closed_form():
    # V = 2, z = (0, x): p1 = sigmoid(x), H = binary entropy.
    xs = np.array([-7.0, -0.5, 0.0, 0.3, 11.0])
    z = np.stack([np.zeros_like(xs), xs], axis=1)
    _, logp, H, _ = O.token_stats(z, np.ones(5, dtype=int), None)
    p1 = 1 / (1 + np.exp(-xs))
    np.testing.assert_allclose(logp, -np.log1p(np.exp(-xs)), atol=1e-14)
    hb = -(p1 * np.log(p1) + (1 - p1) * np.log(1 - p1))
    np.testing.assert_allclose(H, hb, atol=1e-12)


def test_mask_nonfinite_and_bad_id():
    z = np.zeros((4, 8))
    z[2, 3] = np.nan
    z[3, 1] = -np.inf
    mask = np.array([1, 0, 1, 1])
    ids = np.array([9, 0, 1, 1])
    lse, logp, H, flags = O.token_stats(z, ids, mask)
    assert flags & O.FLAG_BAD_ID and flags & O.FLAG_NONFINITE
    assert logp[0] == 0.0 and lse[0] == pytest.approx(math.log(8))
    assert lse[1] == logp[1] == H[1] == 0.0
    assert np.isnan(lse[2]) and np.isnan(H[3])


def test_bf16_widening_is_exact():
    x = torch.randn(1000, dtype=torch.float32).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(O.bf16_bits_to_f64(bits), x.to(torch.float64).numpy())


# --------------------------------------------------------------------------
# a2/a3 discrepancy and aggregates
# --------------------------------------------------------------------------

def test_mu_equals_pi_gives_zero():
    rng = np.random.default_rng(3)
    lp = -rng.exponential(size=40)
    lr, d, seq, grp, batch, flags = O.seq_discrepancy(lp, lp, None, [0, 10, 25, 40], [0, 2, 3])
    assert flags == 0
    assert np.all(lr == 0) and np.all(d == 0)
    assert np.all(grp["Y"] == 0) and batch["Y_mean"] == 0


def test_distance_is_on_probabilities():
    # pi = 0.5, mu = 0.25: d = 0.25 and lr = ln 2 (Eq. distance_metric uses probabilities)
    lr, d, *_ = O.seq_discrepancy([math.log(0.5)], [math.log(0.25)], None, [0, 1], [0, 1])
    assert d[0] == pytest.approx(0.25, abs=1e-15)
    assert lr[0] == pytest.approx(math.log(2), abs=1e-15)


def test_hand_worked_aggregates():
    # Two prompts.  Prompt 0: seq0 (2 tokens), seq1 (all masked), seq2 (3 tokens, one padded).
    # Prompt 1: seq3 (1 token).  Probabilities chosen so that every d is a short decimal.
    pi = [0.50, 0.40, 0.9, 0.9, 0.30, 0.20, 0.10, 0.99, 0.70]
    mu = [0.40, 0.40, 0.1, 0.1, 0.25, 0.30, 0.10, 0.50, 0.60]
    mask = [1, 1, 0, 0, 1, 1, 1, 0, 1]
    so = [0, 2, 4, 8, 9]
    go = [0, 3, 4]
    lr, d, seq, grp, batch, flags = O.seq_discrepancy(np.log(pi), np.log(mu), mask, so, go)
    assert flags == 0
    # by hand: seq0 d = (0.1, 0.0) -> D0 = 0.05 ; seq2 d = (0.05, 0.1, 0.0) -> D2 = 0.05
    # seq3 d = (0.1,) -> D3 = 0.1 ; Y_0 = (0.05 + 0.05) / 2 (seq1 has no valid token) ; Y_1 = 0.1
    np.testing.assert_allclose(d, [0.1, 0, 0, 0, 0.05, 0.1, 0, 0, 0.1], atol=1e-15)
    assert list(seq["n"]) == [2, 0, 3, 1]
    np.testing.assert_allclose(seq["mean_d"], [0.05, 0, 0.05, 0.1], atol=1e-15)
    np.testing.assert_allclose(seq["max_d"], [0.1, 0, 0.1, 0.1], atol=1e-15)
    assert list(grp["n_valid_seqs"]) == [2, 1]
    np.testing.assert_allclose(grp["Y"], [0.05, 0.1], atol=1e-15)
    assert batch["n_groups_valid"] == 2 and batch["n_tokens"] == 6 and batch["n_seqs_valid"] == 3
    np.testing.assert_allclose(batch["Y_mean"], 0.075, atol=1e-15)
    np.testing.assert_allclose(batch["d_mean"], 0.35 / 6, atol=1e-15)
    np.testing.assert_allclose(batch["d_max"], 0.1, atol=1e-15)
    dv = np.array([0.1, 0.0, 0.05, 0.1, 0.0, 0.1])
    np.testing.assert_allclose(batch["d_std"], math.sqrt(np.mean((dv - dv.mean()) ** 2)), atol=1e-15)
    # MIS log-ratio of seq2 = ln(0.3/0.25) + ln(0.2/0.3) + ln(0.1/0.1) = ln(0.8)
    assert seq["sum_lr"][2] == pytest.approx(math.log(0.8), abs=1e-14)


def test_aggregates_as_linear_functional():
    # Y_g = sum_t c_t d_t with c_t = 1/(G_g n_i) on valid tokens: an independent formulation.
    rng = np.random.default_rng(5)
    lengths = [5, 0, 12, 7, 3, 9]
    so = np.concatenate([[0], np.cumsum(lengths)])
    go = [0, 3, 4, 6]
    T = so[-1]
    mask = (rng.random(T) < 0.8).astype(np.uint8)
    pi = -rng.exponential(size=T)
    mu = pi + rng.normal(0, 0.3, size=T)
    _, _, seq, grp, batch, _ = O.seq_discrepancy(pi, mu, mask, so, go)
    for g in range(3):
        seqs = range(go[g], go[g + 1])
        n = {i: int(mask[so[i]:so[i + 1]].sum()) for i in seqs}
        Gg = sum(1 for i in seqs if n[i] > 0)
        acc = []
        for i in seqs:
            for t in range(so[i], so[i + 1]):
                if mask[t] and n[i] > 0:
                    acc.append(abs(math.exp(pi[t]) - math.exp(mu[t])) / (Gg * n[i]))
        assert grp["Y"][g] == pytest.approx(math.fsum(acc), abs=1e-14)


def test_bad_offsets_flagged():
    *_, flags = O.seq_discrepancy(np.zeros(5), np.zeros(5), None, [0, 3, 2, 5], [0, 3])
    assert flags & O.FLAG_BAD_OFFSETS
    *_, flags = O.seq_discrepancy(np.zeros(5), np.zeros(5), None, [0, 3, 4], [0, 2])
    assert flags & O.FLAG_BAD_OFFSETS


# --------------------------------------------------------------------------
# a4 GRPO advantage
# --------------------------------------------------------------------------

@pytest.mark.parametrize("G,k", [(8, 1), (8, 3), (8, 7), (4, 2), (2, 1)])
def test_grpo_binary_closed_form(G, k):
    R = np.array([1.0] * k + [0.0] * (G - k))
    p = O.Params(adv_eps=0.0)
    A = O.grpo_advantage(R, [0, G], p)
    std = math.sqrt(k * (G - k) / (G * (G - 1)))
    np.testing.assert_allclose(A[:k], (1 - k / G) / std, rtol=1e-13)
    np.testing.assert_allclose(A[k:], -(k / G) / std, rtol=1e-13)
    # the epsilon is added to the standard deviation (reading of the A formula under Eq. grpo_objective)
    A = O.grpo_advantage(R, [0, G], O.Params(adv_eps=0.25))
    np.testing.assert_allclose(A[:k], (1 - k / G) / (std + 0.25), rtol=1e-13)
    np.testing.assert_allclose(A[k:], -(k / G) / (std + 0.25), rtol=1e-13)


def test_grpo_matches_scipy_zscore():
    rng = np.random.default_rng(9)
    R = rng.normal(size=24)
    go = [0, 8, 13, 24]
    for ddof in (0, 1):
        A = O.grpo_advantage(R, go, O.Params(adv_eps=0.0, adv_ddof=ddof))
        for g in range(3):
            np.testing.assert_allclose(A[go[g]:go[g + 1]], scipy.stats.zscore(R[go[g]:go[g + 1]], ddof=ddof),
                                       rtol=1e-12)


def test_grpo_equal_rewards_without_epsilon():
    # all-equal rewards with adv_eps = 0: the definition's 0/0 is read as no advantage
    A = O.grpo_advantage(np.array([1.0, 1.0, 1.0, 0.0, 1.0]), [0, 3, 5], O.Params(adv_eps=0.0))
    assert np.all(A[:3] == 0.0)
    np.testing.assert_allclose(A[3:], [-math.sqrt(0.5), math.sqrt(0.5)], rtol=1e-14)   # (0 or 1 - 0.5) / sqrt(0.5)
    # equal rewards whose float64 mean is not exact (found by the property test): still no advantage
    r = 0.9798852880475015
    assert sum([r, r, r]) / 3 != r
    for eps in (0.0, 1e-6):
        assert np.all(O.grpo_advantage(np.array([r, r, r]), [0, 3], O.Params(adv_eps=eps)) == 0.0)


def test_grpo_special_groups():
    R = np.array([0.7, 1.0, 1.0, 1.0, 0.0])
    A = O.grpo_advantage(R, [0, 1, 4, 4, 5], O.Params())
    assert A[0] == 0.7 and A[4] == 0.0          # singletons: mean 0, std 1
    assert np.all(A[1:4] == 0.0)                # all-equal group
    A = O.grpo_advantage(R, [0, 1, 4, 4, 5], O.Params(singleton_rule=O.SINGLETON_ZERO))
    assert A[0] == 0.0


# --------------------------------------------------------------------------
# a5 controller and weights
# --------------------------------------------------------------------------

def _one_token_case(pi, mu, A, Y, X, mode=O.MODE_ACRL, gamma=0.65, C=3.0):
    """A single response with one token, with Y forced through the group stats."""
    lr = np.array([math.log(pi) - math.log(mu)])
    seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([Y]), "sum_lr": lr.copy()}
    grp = {"Y": np.array([Y]), "n_valid_seqs": np.array([1])}
    batch = {"Y_sum": Y, "Y_mean": Y, "n_groups_valid": 1}
    p = O.Params(gamma=gamma, C=C, mode=mode, X_init=X)
    st = O.controller_init(p)
    return O.controller_step(st, p, lr, None, [0, 1], [0, 1], seq, grp, batch, np.array([A]))


def _read_quadrants():
    rows = []
    with open(os.path.join(GOLDEN, "acrl_quadrants.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append(line.split())
    assert len(rows) == 8
    return rows


@pytest.mark.parametrize("row", _read_quadrants(), ids=lambda r: f"{r[0]}-{r[1]}")
def test_quadrant_sign_table(row):
    regime, _, sA, pvm, salpha, rho_vs = row[:6]
    X = 0.013
    Y = 0.02 if regime == "Y>X" else 0.005
    A = 1.0 if sA == "+" else -1.0
    pi, mu = (0.3, 0.5) if pvm == "<" else (0.5, 0.3)
    w, alpha, *_ = _one_token_case(pi, mu, A, Y, X)
    assert (alpha[0] > 0) == (salpha == "+") and alpha[0] != 0
    rho = (pi / mu) ** alpha[0]
    assert (w[0] > 1) == (rho_vs == ">")
    assert w[0] == pytest.approx(min(rho, 3.0), rel=1e-14)


def test_controller_special_cases():
    w, alpha, *_ = _one_token_case(0.2, 0.4, 1.0, 0.013, 0.013)   # Y = X
    assert alpha[0] == 0.0 and w[0] == 1.0
    w, alpha, *_ = _one_token_case(0.2, 0.4, 0.0, 0.05, 0.013)    # A = 0
    assert alpha[0] == 0.0 and w[0] == 1.0
    w, alpha, *_ = _one_token_case(0.3, 0.3, 1.0, 0.05, 0.013)    # mu = pi
    assert w[0] == 1.0
    # alpha = gamma (1 - Y/X) by hand: gamma 0.5, Y = 0.026, X = 0.013 -> alpha = -0.5
    w, alpha, *_ = _one_token_case(0.25, 0.5, 2.0, 0.026, 0.013, gamma=0.5)
    assert alpha[0] == pytest.approx(-0.5, abs=1e-15)
    assert w[0] == pytest.approx(math.sqrt(2.0), rel=1e-14)


def test_tis_and_mis_thresholds():
    w, *_ = _one_token_case(2.9, 1.0, 1.0, 0, 1, mode=O.MODE_TIS)
    assert w[0] == pytest.approx(2.9, rel=1e-14)
    w, _, _, info, _ = _one_token_case(3.1, 1.0, 1.0, 0, 1, mode=O.MODE_TIS)
    assert w[0] == pytest.approx(3.0, rel=1e-14) and info["trunc_frac"] == 1.0
    w, *_ = _one_token_case(2.9, 1.0, 1.0, 0, 1, mode=O.MODE_MIS)
    assert w[0] == pytest.approx(2.9, rel=1e-14)
    w, _, _, info, _ = _one_token_case(3.1, 1.0, 1.0, 0, 1, mode=O.MODE_MIS)
    assert w[0] == 0.0 and info["trunc_frac"] == 1.0
    w, *_ = _one_token_case(3.1, 1.0, -1.0, 0, 1, mode=O.MODE_NONE)
    assert w[0] == 1.0


def test_mis_sequence_ratio_is_product():
    # rho_i = prod_t pi/mu over the valid tokens of the response (Eq. MIS)
    # (a product away from 1, so that a mean of the log-ratios or a single token's ratio cannot pass)
    pi = np.array([0.5, 0.2, 0.9, 0.3])
    mu = np.array([0.4, 0.5, 0.6, 0.1])
    mask = np.array([1, 1, 1, 0])
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(np.log(pi), np.log(mu), mask, [0, 4], [0, 1])
    p = O.Params(mode=O.MODE_MIS, X_init=1.0)
    w, *_ = O.controller_step(O.controller_init(p), p, lr, mask, [0, 4], [0, 1], seq, grp, batch, [1.0])
    prod = (0.5 / 0.4) * (0.2 / 0.5) * (0.9 / 0.6)   # 0.75, the masked token left out
    np.testing.assert_allclose(w, [prod, prod, prod, 0.0], rtol=1e-14)


def test_calibration_then_frozen():
    rng = np.random.default_rng(11)
    p = O.Params()
    st = O.controller_init(p)
    so, go = [0, 4, 9, 15, 20], [0, 2, 4]
    Xs = []
    for k in range(50):
        pi = -rng.exponential(size=20)
        mu = pi + rng.normal(0, 0.1, size=20)
        lr, d, seq, grp, batch, _ = O.seq_discrepancy(pi, mu, None, so, go)
        if k == 0:
            X0 = (grp["Y"][0] + grp["Y"][1]) / 2
        _, _, st, info, _ = O.controller_step(st, p, lr, None, so, go, seq, grp, batch, np.ones(4))
        Xs.append(st.X)
    assert st.calibrated and st.step == 50
    assert Xs[0] == X0 and all(x == X0 for x in Xs)


def test_multi_step_calibration():
    p = O.Params(calib_steps=3)
    st = O.controller_init(p)
    Ys = [0.01, 0.03, 0.02]
    for k, Y in enumerate(Ys):
        lr = np.array([0.5])
        seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([Y]), "sum_lr": lr}
        grp = {"Y": np.array([Y]), "n_valid_seqs": np.array([1])}
        batch = {"Y_sum": Y, "Y_mean": Y, "n_groups_valid": 1}
        w, alpha, st, info, _ = O.controller_step(st, p, lr, None, [0, 1], [0, 1], seq, grp, batch, [1.0])
        if k < 2:
            assert alpha[0] == 0.0 and w[0] == 1.0 and not st.calibrated
    assert st.calibrated and st.X == pytest.approx(0.02, abs=1e-15)


def _lr_case(lr_value, A, mode=O.MODE_ACRL, Y=0.026, X=0.013):
    lr = np.array([lr_value])
    seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([Y]), "sum_lr": lr.copy()}
    grp = {"Y": np.array([Y]), "n_valid_seqs": np.array([1])}
    batch = {"Y_sum": Y, "Y_mean": Y, "n_groups_valid": 1}
    p = O.Params(mode=mode, X_init=X)
    return O.controller_step(O.controller_init(p), p, lr, None, [0, 1], [0, 1], seq, grp, batch, np.array([A]))


def test_infinite_and_nan_log_ratios():
    # mu = 0 on a sampled token: lr = +inf.  rho^0 = 1 (A = 0 gives alpha = 0), TIS truncates at C, an
    # exponent of either sign follows min(rho^alpha, C) (C, or 0); MIS truncates the sequence
    assert _lr_case(math.inf, 0.0)[0][0] == 1.0
    assert _lr_case(math.inf, 1.0, mode=O.MODE_TIS)[0][0] == pytest.approx(3.0, rel=1e-15)
    assert _lr_case(math.inf, -1.0)[0][0] == pytest.approx(3.0, rel=1e-15)  # Y > X, A < 0: alpha > 0
    assert _lr_case(math.inf, 1.0)[0][0] == 0.0           # Y > X, A > 0: alpha < 0
    assert _lr_case(math.inf, 1.0, mode=O.MODE_MIS)[0][0] == 0.0
    # a NaN log-prob: the token's weight is 0 and the discrepancy pass flags it
    for mode in (O.MODE_ACRL, O.MODE_TIS, O.MODE_MIS):
        assert _lr_case(math.nan, 1.0, mode=mode)[0][0] == 0.0
    *_, f = O.seq_discrepancy(np.array([-1.0, -2.0]), np.array([-1.5, math.nan]), None, [0, 2], [0, 1])
    assert f & O.FLAG_NONFINITE
    lr, d, *_, f = O.seq_discrepancy(np.array([-1.0]), np.array([-math.inf]), None, [0, 1], [0, 1])
    assert f == 0 and lr[0] == math.inf and d[0] == pytest.approx(math.exp(-1.0), rel=1e-15)


def test_calibration_averages_prompts_across_batches():
    # X is the mean of Y_g over every prompt of the calibration batches (Sec. 4.1): batches of 1 and 3 prompts
    # give (0.01 + 3 x 0.03) / 4 = 0.025, not the mean of the two batch means (0.02)
    p = O.Params(calib_steps=2)
    st = O.controller_init(p)
    for Ys in ([0.01], [0.03, 0.03, 0.03]):
        G = len(Ys)
        lr = np.full(G, 0.5)
        seq = {"n": np.ones(G, dtype=np.int64), "group": np.arange(G), "mean_d": np.array(Ys), "sum_lr": lr}
        grp = {"Y": np.array(Ys), "n_valid_seqs": np.ones(G, dtype=np.int64)}
        batch = {"Y_sum": sum(Ys), "Y_mean": sum(Ys) / G, "n_groups_valid": G}
        offs = list(range(G + 1))
        _, _, st, _, _ = O.controller_step(st, p, lr, None, offs, offs, seq, grp, batch, np.ones(G))
    assert st.calibrated and st.X == pytest.approx(0.025, abs=1e-15)


def test_nonpositive_X_flag_and_fixed_point():
    # mu = pi everywhere: d = 0, X calibrates to 0, alpha := 0 and every weight is 1
    rng = np.random.default_rng(2)
    lp = -rng.exponential(size=12)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(lp, lp, None, [0, 5, 12], [0, 2])
    p = O.Params()
    w, alpha, st, info, flags = O.controller_step(O.controller_init(p), p, lr, None, [0, 5, 12], [0, 2],
                                                  seq, grp, batch, [1.0, -1.0])
    assert flags & O.FLAG_X_NONPOS
    assert np.all(w == 1.0) and np.all(alpha == 0.0) and st.X == 0.0


def test_y_granularity_options():
    pi = np.log([0.5, 0.5, 0.5, 0.5])
    mu = np.log([0.4, 0.4, 0.3, 0.3])   # d: seq0 0.1, seq1 0.2
    so, go = [0, 2, 4], [0, 2]
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(pi, mu, None, so, go)
    A = [1.0, 1.0]
    out = {}
    for gran in (O.Y_GROUP, O.Y_SEQUENCE, O.Y_BATCH):
        p = O.Params(gamma=1.0, X_init=0.1, y_gran=gran)
        _, alpha, *_ = O.controller_step(O.controller_init(p), p, lr, None, so, go, seq, grp, batch, A)
        out[gran] = alpha
    np.testing.assert_allclose(out[O.Y_GROUP], [-0.5, -0.5], atol=1e-14)     # Y = 0.15
    np.testing.assert_allclose(out[O.Y_SEQUENCE], [0.0, -1.0], atol=1e-14)   # Y = 0.1, 0.2
    np.testing.assert_allclose(out[O.Y_BATCH], [-0.5, -0.5], atol=1e-14)


# --------------------------------------------------------------------------
# a6 loss and gradient
# --------------------------------------------------------------------------

def _fixture(rng, V=9, with_old=True):
    lengths = [3, 2, 4, 1]
    so = np.concatenate([[0], np.cumsum(lengths)])
    go = [0, 2, 4]
    T = int(so[-1])
    z = rng.normal(0, 1.5, size=(T, V))
    ids = rng.integers(0, V, size=T)
    mask = np.array([1, 1, 0, 1, 1, 1, 1, 1, 1, 1])
    lse, logp, H, _ = O.token_stats(z, ids, mask)
    mu = logp + rng.normal(0, 0.2, size=T)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(logp, mu, mask, so, go, H)
    adv = np.array([0.8, -1.3, 0.0, 2.0])
    w = np.where(mask, rng.uniform(0.5, 2.0, size=T), 0.0)
    old = logp + rng.normal(0, 0.4, size=T) if with_old else None
    return dict(z=z, ids=ids, mask=mask, lse=lse, old=old, adv=adv, w=w, so=so, go=go, seq=seq, grp=grp,
                batch=batch)


def _torch_loss(zt, f, params):
    """The loss written with torch ops; autograd differentiates it."""
    logq = torch.log_softmax(zt, dim=1)
    logp = logq[torch.arange(zt.shape[0]), torch.as_tensor(f["ids"])]
    if f["old"] is None:
        r = torch.exp(logp - logp.detach())    # theta = theta_old: r = 1 in value, gradient r * dlogp
    else:
        r = torch.exp(logp - torch.as_tensor(f["old"]))
    total = torch.zeros((), dtype=torch.float64)
    so = f["so"]
    for i in range(len(so) - 1):
        g = int(f["seq"]["group"][i])
        n = f["seq"]["n"][i]
        for t in range(so[i], so[i + 1]):
            if not f["mask"][t]:
                continue
            norm = f["batch"]["n_groups_valid"] * f["grp"]["n_valid_seqs"][g] * n
            A = f["adv"][i]
            surr = torch.minimum(r[t] * A, torch.clamp(r[t], 1 - params.clip_eps, 1 + params.clip_eps) * A)
            total = total - f["w"][t] * surr / norm
            if params.entropy_coeff:
                ent = -(torch.softmax(zt[t], 0) * logq[t]).sum()
                total = total - params.entropy_coeff * ent / norm
    return total


@pytest.mark.parametrize("beta", [0.0, 0.05])
@pytest.mark.parametrize("with_old", [False, True])
def test_gradient_matches_autograd(with_old, beta):
    rng = np.random.default_rng(21 + with_old)
    f = _fixture(rng, with_old=with_old)
    p = O.Params(entropy_coeff=beta)
    grad, tl, loss = O.loss_grad_logits(f["z"], f["ids"], f["mask"], None, f["old"], f["adv"], f["w"], f["so"],
                                        f["seq"], f["grp"], f["batch"], p)
    zt = torch.tensor(f["z"], dtype=torch.float64, requires_grad=True)
    L = _torch_loss(zt, f, p)
    L.backward()
    np.testing.assert_allclose(grad, zt.grad.numpy(), atol=1e-14)
    assert loss == pytest.approx(float(L.detach()), abs=1e-14)


@pytest.mark.parametrize("recompute", [False, True])
def test_gradient_undefined_rows(recompute):
    """Readings c17 and c18 in the gradient.  A live row whose log-sum-exp or
    log-prob is not finite (a NaN or an infinity among its logits), or whose
    old log-prob is NaN, has no defined surrogate: its token loss and its whole
    gradient row are NaN, and so is the loss.  A row with a zero weighted
    advantage, or a masked row, stays a zero row with token loss 0 whatever
    its logits hold.  Every other row is exactly what it is without them."""
    rng = np.random.default_rng(41)
    f = _fixture(rng, with_old=True)
    p = O.Params()

    def run(z, old):
        lse = None if recompute else O.token_stats(z, f["ids"], f["mask"])[0]
        return O.loss_grad_logits(z, f["ids"], f["mask"], lse, old, f["adv"], f["w"], f["so"], f["seq"], f["grp"],
                                  f["batch"], p)

    g0, tl0, loss0 = run(f["z"], f["old"])
    assert np.isfinite(loss0) and np.all(np.isfinite(g0))
    z, old = f["z"].copy(), f["old"].copy()
    z[3, 1] = np.nan        # live (advantage -1.3)
    z[4, 2] = np.inf        # live
    old[9] = np.nan         # live (advantage 2.0)
    z[6, 0] = np.nan        # advantage 0: a zero row, never read
    z[2, :] = np.nan        # masked
    g, tl, loss = run(z, old)
    bad = [3, 4, 9]
    assert np.all(np.isnan(g[bad])) and np.all(np.isnan(tl[bad])) and np.isnan(loss)
    assert np.all(g[[2, 6]] == 0.0) and tl[2] == 0.0 and tl[6] == 0.0
    good = [t for t in range(len(tl)) if t not in bad]
    assert np.array_equal(g[good], g0[good]) and np.array_equal(tl[good], tl0[good])


@pytest.mark.parametrize("beta", [0.0, 0.3])
def test_gradient_central_differences(beta):
    rng = np.random.default_rng(33)
    f = _fixture(rng, V=6, with_old=True)
    p = O.Params(entropy_coeff=beta)

    def L(z):
        return O.loss_grad_logits(z, f["ids"], f["mask"], None, f["old"], f["adv"], f["w"], f["so"], f["seq"],
                                  f["grp"], f["batch"], p)[2]

    grad = O.loss_grad_logits(f["z"], f["ids"], f["mask"], None, f["old"], f["adv"], f["w"], f["so"], f["seq"],
                              f["grp"], f["batch"], p)[0]
    h = 1e-6
    num = np.zeros_like(f["z"])
    for t in range(f["z"].shape[0]):
        for j in range(f["z"].shape[1]):
            zp = f["z"].copy()
            zm = f["z"].copy()
            zp[t, j] += h
            zm[t, j] -= h
            num[t, j] = (L(zp) - L(zm)) / (2 * h)
    np.testing.assert_allclose(grad, num, rtol=1e-6, atol=1e-9)


def test_on_policy_loss_by_hand_and_invariants():
    # r = 1: loss = -sum_t w_t A_i / (Q_eff G_g n_i).  Two prompts, seqs of 2 and 1 tokens + 1 token.
    V = 5
    z = np.zeros((4, V))
    ids = np.array([0, 1, 2, 3])
    so, go = [0, 2, 3, 4], [0, 2, 3]
    mask = np.ones(4, dtype=np.uint8)
    seq = {"n": np.array([2, 1, 1]), "group": np.array([0, 0, 1])}
    grp = {"n_valid_seqs": np.array([2, 1])}
    batch = {"n_groups_valid": 2, "n_tokens": 4}
    adv = np.array([1.0, -2.0, 0.5])
    w = np.array([1.0, 2.0, 0.5, 3.0])
    grad, tl, loss = O.loss_grad_logits(z, ids, mask, None, None, adv, w, so, seq, grp, batch, O.Params())
    by_hand = -(1.0 * 1.0 / 8 + 2.0 * 1.0 / 8 + 0.5 * -2.0 / 4 + 3.0 * 0.5 / 2)
    assert loss == pytest.approx(by_hand, abs=1e-15)
    np.testing.assert_allclose(grad.sum(axis=1), 0.0, atol=1e-15)   # sum_j (p_j - 1[j=a]) = 0
    # uniform row: grad[t, j] = coef (1/V - 1[j = a])
    assert grad[0, 0] == pytest.approx(1.0 / 8 * (1 / V - 1), abs=1e-15)
    assert grad[0, 1] == pytest.approx(1.0 / 8 * (1 / V), abs=1e-15)
    # TOKEN_MEAN aggregation divides by the valid-token count instead
    _, _, loss_tm = O.loss_grad_logits(z, ids, mask, None, None, adv, w, so, seq, grp, batch,
                                       O.Params(agg=O.AGG_TOKEN_MEAN))
    assert loss_tm == pytest.approx(-(1.0 + 2.0 - 1.0 + 1.5) / 4, abs=1e-15)


def test_clip_gate():
    # A > 0 and r > 1 + eps: clipped branch, no gradient; A < 0 and r < 1 - eps likewise.
    V = 4
    z = np.zeros((2, V))
    ids = np.array([0, 0])
    lp = math.log(0.25)
    old = np.array([lp - 0.5, lp + 0.5])        # r = e^0.5 > 1.2 ; r = e^-0.5 < 0.8
    seq = {"n": np.array([1, 1]), "group": np.array([0, 0])}
    grp = {"n_valid_seqs": np.array([2])}
    batch = {"n_groups_valid": 1, "n_tokens": 2}
    for A, zero_row in (([1.0, 1.0], 0), ([-1.0, -1.0], 1)):
        grad, tl, loss = O.loss_grad_logits(z, ids, None, None, old, np.array(A), np.ones(2), [0, 1, 2], seq, grp,
                                            batch, O.Params())
        assert np.all(grad[zero_row] == 0) and np.any(grad[1 - zero_row] != 0)


def test_full_step_mu_equals_pi_fixed_point():
    rng = np.random.default_rng(8)
    T, V = 12, 16
    z = rng.normal(size=(T, V))
    ids = rng.integers(0, V, size=T)
    _, logp, _, _ = O.token_stats(z, ids, None)
    res = O.step(z, ids, None, logp, np.array([1.0, 0.0, 1.0]), [0, 4, 8, 12], [0, 3], O.Params())
    assert np.all(res.lr == 0) and np.all(res.weight == 1.0)
    assert res.state.X == 0.0 and res.flags & O.FLAG_X_NONPOS


@pytest.mark.parametrize("with_old", [False, True])
def test_coefficients_and_surrogate_agree_with_gradient(with_old):
    # coef_t (p - onehot) r g must reproduce the autograd-pinned gradient, and the
    # O(T) surrogate loss must equal the loss of loss_grad_logits.
    rng = np.random.default_rng(44 + with_old)
    f = _fixture(rng, with_old=with_old)
    p = O.Params()
    grad, tl, loss = O.loss_grad_logits(f["z"], f["ids"], f["mask"], None, f["old"], f["adv"], f["w"], f["so"],
                                        f["seq"], f["grp"], f["batch"], p)
    coef = O.loss_coefficients(f["w"], f["adv"], f["mask"], f["so"], f["seq"], f["grp"], f["batch"], p)
    lse, logp, _, _ = O.token_stats(f["z"], f["ids"], f["mask"])
    tl2, loss2 = O.surrogate_loss(logp, f["old"], f["adv"], f["w"], f["mask"], f["so"], f["seq"], f["grp"],
                                  f["batch"], p)
    assert loss2 == pytest.approx(loss, abs=1e-14)
    np.testing.assert_allclose(tl2, tl, atol=1e-15)
    for t in range(len(coef)):
        r = 1.0 if f["old"] is None else math.exp(logp[t] - f["old"][t])
        gate = (coef[t] >= 0 and r <= 1.2) or (coef[t] < 0 and r >= 0.8)
        pr = np.exp(f["z"][t] - lse[t])
        pr[f["ids"][t]] -= 1.0
        np.testing.assert_allclose(grad[t], coef[t] * r * gate * pr, atol=1e-15)


def test_entropy_bonus_by_hand():
    # uniform rows: H = ln V, so each valid token adds -beta ln V / norm to the loss
    V = 6
    z = np.zeros((3, V))
    ids = np.array([0, 1, 2])
    seq = {"n": np.array([2, 1]), "group": np.array([0, 0])}
    grp = {"n_valid_seqs": np.array([2])}
    batch = {"n_groups_valid": 1, "n_tokens": 3}
    adv = np.array([0.0, 0.0])                     # no policy term: only the bonus
    p = O.Params(entropy_coeff=0.1)
    grad, tl, loss = O.loss_grad_logits(z, ids, None, None, None, adv, np.ones(3), [0, 2, 3], seq, grp, batch, p)
    assert loss == pytest.approx(-0.1 * math.log(V) * (1 / 4 + 1 / 4 + 1 / 2), abs=1e-15)
    # at the uniform distribution the entropy is maximal: its gradient vanishes
    np.testing.assert_allclose(grad, 0.0, atol=1e-16)
    beta_t = O.entropy_coefficients(None, [0, 2, 3], seq, grp, batch, p)
    np.testing.assert_allclose(beta_t, [0.1 / 4, 0.1 / 4, 0.1 / 2], rtol=1e-15)


@pytest.mark.parametrize("row", _read_quadrants(), ids=lambda r: f"{r[0]}-{r[1]}")
def test_continuous_reduction_always_reduces(row):
    # Sec. 5.5: alpha = -1 where A > 0 and +1 where A < 0 whatever Y and X are, so every
    # quadrant follows the Y > X (decrease) row of the sign table.
    _, quad, sA, pvm = row[:4]
    table = {r[1]: r for r in _read_quadrants() if r[0] == "Y>X"}
    A = 1.0 if sA == "+" else -1.0
    pi, mu = (0.3, 0.5) if pvm == "<" else (0.5, 0.3)
    for Y in (0.005, 0.02):
        w, alpha, *_ = _one_token_case(pi, mu, A, Y, 0.013, mode=O.MODE_ACRL_CONTINUOUS)
        assert alpha[0] == -A
        assert (w[0] > 1) == (table[quad][5] == ">")
        assert w[0] == pytest.approx(min((pi / mu) ** -A, 3.0), rel=1e-14)


def test_continuous_reduction_kappa():
    w, alpha, *_ = _one_token_case(0.2, 0.4, -1.0, 0.0, 0.013, mode=O.MODE_ACRL_CONTINUOUS)
    assert alpha[0] == 1.0 and w[0] == pytest.approx(0.5, rel=1e-14)
    p = O.Params(mode=O.MODE_ACRL_CONTINUOUS, kappa=3.0, X_init=0.013)
    lr = np.array([math.log(0.5)])
    seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([0.0]), "sum_lr": lr}
    grp = {"Y": np.array([0.0]), "n_valid_seqs": np.array([1])}
    batch = {"Y_sum": 0.0, "Y_mean": 0.0, "n_groups_valid": 1}
    w, alpha, *_ = O.controller_step(O.controller_init(p), p, lr, None, [0, 1], [0, 1], seq, grp, batch, [2.0])
    assert alpha[0] == -3.0 and w[0] == pytest.approx(3.0, rel=1e-14)   # (1/2)^-3 = 8, truncated at C = 3


def test_fallback_to_grpo():
    # Y < X: plain GRPO (w = 1); Y > X: the ACRL weight
    w, alpha, *_ = _one_token_case(0.2, 0.4, 1.0, 0.005, 0.013, mode=O.MODE_ACRL_FALLBACK)
    assert alpha[0] == 0.0 and w[0] == 1.0
    w, alpha, *_ = _one_token_case(0.2, 0.4, 1.0, 0.026, 0.013, mode=O.MODE_ACRL_FALLBACK, gamma=0.5)
    assert alpha[0] == pytest.approx(-0.5, abs=1e-15) and w[0] == pytest.approx(math.sqrt(2), rel=1e-14)


def test_moving_average_X_by_hand():
    # X frozen by default; with x_ema = 0.5 each later step moves X halfway to that step's Y
    p = O.Params(x_ema=0.5)
    st = O.controller_init(p)
    Xs = []
    for Y in (0.02, 0.04, 0.01):
        lr = np.array([0.1])
        seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([Y]), "sum_lr": lr}
        grp = {"Y": np.array([Y]), "n_valid_seqs": np.array([1])}
        batch = {"Y_sum": Y, "Y_mean": Y, "n_groups_valid": 1}
        _, _, st, info, _ = O.controller_step(st, p, lr, None, [0, 1], [0, 1], seq, grp, batch, [1.0])
        Xs.append((info["X"], st.X))
    # step 0 calibrates X = 0.02 (no update on that step); step 1 uses 0.02 then moves to 0.03; step 2 uses 0.03
    assert Xs[0] == (pytest.approx(0.02), pytest.approx(0.02))
    assert Xs[1] == (pytest.approx(0.02), pytest.approx(0.03))
    assert Xs[2] == (pytest.approx(0.03), pytest.approx(0.02))


def test_round_bf16_matches_library_and_ties():
    rng = np.random.default_rng(12)
    x = rng.normal(0, 3, size=20000).astype(np.float32).astype(np.float64)
    ref = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x), ref)
    # ties go to the even mantissa: 1 + 2^-8 -> 1, 1 + 3 * 2^-8 -> 1 + 2^-6 ... (spacing 2^-7 in [1, 2))
    assert O.round_bf16(1 + 2 ** -8) == 1.0
    assert O.round_bf16(1 + 3 * 2 ** -8) == 1 + 2 ** -6
    assert O.round_bf16(-(1 + 2 ** -8)) == -1.0
    assert O.round_bf16(1 + 2 ** -8 + 2 ** -30) == 1 + 2 ** -7


def test_lmhead_logits_small():
    rng = np.random.default_rng(13)
    H = O.round_bf16(rng.normal(size=(5, 40)))
    W = O.round_bf16(rng.normal(0, 0.2, size=(7, 40)))
    z = O.lmhead_logits(H, W)
    for i in range(5):
        for j in range(7):
            exact = math.fsum(H[i, k] * W[j, k] for k in range(40))
            assert z[i, j] == O.round_bf16(exact)
