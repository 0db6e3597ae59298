"""Property-based checks of the oracle (CPU): invariants that hold for any
input the generators draw, on top of the fixed pins of test_oracle_pins.py.
Each property follows from the definitions, not from the oracle's own code:
shift invariance and bounds of the log-softmax statistics, zero row sums of
the on-policy gradient, centred and unit-std GRPO advantages, and weights
inside (0, C] that move the right way for the sign table of Sec. 4.2."""

import math

import numpy as np
import pytest

hyp = pytest.importorskip("hypothesis")
from hypothesis import given, settings  # noqa: E402
from hypothesis import strategies as st  # noqa: E402

import oracle as O  # noqa: E402

# derandomized: the same examples every run, so that the suite's outcome does not depend on the run
SETTINGS = settings(max_examples=60, deadline=None, derandomize=True)


@st.composite
def logit_rows(draw, max_rows=4, max_v=40):
    T = draw(st.integers(1, max_rows))
    V = draw(st.integers(1, max_v))
    z = np.array(draw(st.lists(st.floats(-30, 30, allow_nan=False), min_size=T * V, max_size=T * V)))
    ids = np.array(draw(st.lists(st.integers(0, V - 1), min_size=T, max_size=T)))
    return z.reshape(T, V), ids


@SETTINGS
@given(logit_rows(), st.floats(-50, 50, allow_nan=False))
def test_token_stats_shift_invariance_and_bounds(zi, c):
    z, ids = zi
    V = z.shape[1]
    lse, logp, H, f = O.token_stats(z, ids, None)
    lse2, logp2, H2, _ = O.token_stats(z + c, ids, None)
    assert f == 0
    np.testing.assert_allclose(lse2, lse + c, rtol=0, atol=1e-9 * (1 + abs(c) + float(np.abs(lse).max())))
    np.testing.assert_allclose(logp2, logp, rtol=0, atol=1e-9 * (1 + abs(c)))
    np.testing.assert_allclose(H2, H, rtol=0, atol=1e-9 * (1 + abs(c)))
    assert np.all(logp <= 1e-12)
    assert np.all(H >= -1e-12) and np.all(H <= math.log(V) + 1e-9)


@SETTINGS
@given(logit_rows(max_v=24))
def test_token_stats_matches_bruteforce_on_random_rows(zi):
    z, ids = zi
    lse, logp, H, _ = O.token_stats(z, ids, None)
    blse, blogp, bH = O.token_stats_bruteforce(z, ids)
    np.testing.assert_allclose(lse, blse, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(logp, blogp, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(H, bH, rtol=1e-9, atol=1e-12)


@SETTINGS
@given(logit_rows(max_v=30), st.floats(-2, 2, allow_nan=False))
def test_on_policy_gradient_rows_sum_to_zero(zi, A):
    # sum_j (p_j - 1[j = a]) = 0 for every row, so every gradient row sums to 0
    z, ids = zi
    T = len(ids)
    lse, *_ = O.token_stats(z, ids, None)
    seq = {"n": np.array([T]), "group": np.array([0])}
    grp = {"n_valid_seqs": np.array([1])}
    batch = {"n_groups_valid": 1, "n_tokens": T}
    grad, tl, loss = O.loss_grad_logits(z, ids, None, lse, None, np.array([A]), np.ones(T), [0, T], seq, grp, batch,
                                        O.Params())
    np.testing.assert_allclose(grad.sum(axis=1), 0.0, atol=1e-12 * (1 + abs(A)))
    # and the sampled column carries the only negative entries when A > 0
    if A > 0:
        for t in range(T):
            row = np.delete(grad[t], ids[t])
            assert np.all(row >= 0) and grad[t, ids[t]] <= 0


@SETTINGS
@given(st.lists(st.lists(st.floats(0, 1, allow_nan=False), min_size=1, max_size=9), min_size=1, max_size=5))
def test_grpo_advantages_centred_with_unit_std(groups):
    R = np.concatenate([np.array(g) for g in groups])
    go = np.cumsum([0] + [len(g) for g in groups])
    p = O.Params(adv_eps=0.0)
    A = O.grpo_advantage(R, go, p)
    for g in range(len(groups)):
        a, r = A[go[g]:go[g + 1]], R[go[g]:go[g + 1]]
        if len(r) == 1:
            assert a[0] == r[0]                          # mean 0, std 1 for a lone response
        elif np.ptp(r) == 0:
            assert np.all(a == 0.0)                      # equal rewards: no advantage
        elif np.ptp(r) > 1e-9:
            assert abs(a.sum()) <= 1e-9 * len(a)
            assert np.std(a, ddof=1) == pytest.approx(1.0, rel=1e-9)


@SETTINGS
@given(st.floats(0.02, 0.98), st.floats(0.02, 0.98), st.sampled_from([-1.0, 1.0]), st.floats(0.001, 0.2),
       st.floats(0.001, 0.2), st.floats(0.1, 2.0))
def test_acrl_weight_bounds_and_direction(pi, mu, A, Y, X, gamma):
    # w = min((pi/mu)^alpha, C) lies in (0, C] (0 only by float64 underflow); alpha = gamma sign(A) (1 - Y/X), and the weight is above 1
    # exactly when alpha and log(pi/mu) have the same sign (the eight cases of the Sec. 4.2 table)
    lr = np.array([math.log(pi) - math.log(mu)])
    seq = {"n": np.array([1]), "group": np.array([0]), "mean_d": np.array([Y]), "sum_lr": lr}
    grp = {"Y": np.array([Y]), "n_valid_seqs": np.array([1])}
    batch = {"Y_sum": Y, "Y_mean": Y, "n_groups_valid": 1}
    p = O.Params(X_init=X, gamma=gamma)
    w, alpha, *_ = O.controller_step(O.controller_init(p), p, lr, None, [0, 1], [0, 1], seq, grp, batch, [A])
    assert 0.0 <= w[0] <= p.C * (1 + 1e-15)
    assert alpha[0] == pytest.approx(gamma * A * (1 - Y / X), rel=1e-12, abs=1e-15)
    if alpha[0] * lr[0] > -700.0:   # rho^alpha itself is positive; only a float64 underflow can make it 0
        assert w[0] > 0.0
    if abs(alpha[0] * lr[0]) > 1e-12 and w[0] < p.C:   # below that, rho^alpha rounds to 1 in float64
        assert (w[0] > 1) == ((alpha[0] > 0) == (pi > mu))
