"""Float64 CPU oracle for the ACRL vocabulary-wide hot path.

TEST INFRASTRUCTURE ONLY.  This module exists so that the CUDA path can be
checked against a plain, slow, obviously correct statement of what the paper
defines.  Only the test-suite, the smoke check and the CPU-baseline leg of the
benchmark may import it; the library and its Python binding never do.  It
shares no code, header, constant table or helper with the CUDA path and
imports nothing from it.

Paper: "ACRL: Adaptive Control of Training-Inference Discrepancy for Stable
Reinforcement Learning" (arXiv 2607.24062).  Every function below cites the
passage it follows.  Everything is computed in float64 with numpy; bf16 logits
are widened to float64 exactly (bf16 is a subset of float64).

Where the paper is silent the oracle takes these readings (they are also the
readings of the CUDA path; each is listed with its reason in the design notes):
  * d is an absolute difference of probabilities, not of log-probabilities
    (Eq. distance_metric, Sec. 4.1).
  * Y defaults to the group form (1/G) sum_i (1/|a_i|) sum_t d, literally the
    formula after Eq. ACRL; per-sequence and whole-batch forms are options.
  * Sequences with no valid token are left out of Y_g and of G_g; a group with
    no valid sequence is left out of the prompt count.
  * GRPO std uses ddof=1 plus adv_eps; a group of one response gets mean 0 and
    std 1 (so A = R) unless the ZERO rule is chosen; a group whose rewards are
    all equal gets A = 0 (decided on the rewards themselves).
  * sign(0) = 0, so A = 0 gives alpha = 0 and rho = 1.
  * min(rho, C) is evaluated as exp(min(alpha*lr, ln C)); the MIS indicator
    1{rho_i <= C} as S_i <= ln C.
  * X is the mean of Y_g over the prompts of the first `calib_steps` batches
    (Sec. 4.1: fixed before training; Sec. 5.1 takes it from step 0), then
    frozen.  If X <= 0 the controller sets alpha = 0 and raises a flag.
  * The clip tie r = 1 +/- eps keeps the unclipped branch.
  * Masked tokens contribute nothing: their outputs are 0 and their gradient
    row is 0.  A row whose coefficient is 0 has a zero gradient row.
  * Any non-finite logit in a valid row makes that row's lse/logp/entropy NaN
    and sets a flag; a sampled id outside [0, V) gives logp = 0, a zero
    gradient row and a flag.  In the gradient, a live row whose log-sum-exp
    or log-prob is not finite, or whose old log-prob is NaN, gets a NaN token
    loss and a NaN gradient row (and the call sets the flag).
  * A log-ratio of +inf (mu = 0 on the sampled token) follows min(rho^alpha, C)
    with rho^0 = 1; a NaN log-ratio gets weight 0 and sets a flag.

Parity status: every function here is pinned by tests that do not re-use its
own formulas (brute force, closed forms, invariants, finite differences and
the sign table of Sec. 4.2).  The paper prints no worked numeric example, so no
function is pinned to a number the paper prints.
"""

from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# Weight modes (Sec. 2.2 TIS / MIS, Sec. 4.1 ACRL, plain GRPO) and the two
# one-sided ablations of Sec. 5.5.
MODE_NONE, MODE_TIS, MODE_MIS, MODE_ACRL = 0, 1, 2, 3
MODE_ACRL_CONTINUOUS, MODE_ACRL_FALLBACK = 4, 5
# Granularity of the current discrepancy Y.
Y_GROUP, Y_SEQUENCE, Y_BATCH = 0, 1, 2
# Loss aggregation.
AGG_SEQ_MEAN_TOKEN_MEAN, AGG_TOKEN_MEAN = 0, 1
# GRPO rule for a group with a single response.
SINGLETON_MEAN0_STD1, SINGLETON_ZERO = 0, 1

# Data-dependent error bits (the oracle's own copy of the library's meaning).
FLAG_BAD_ID = 1
FLAG_NONFINITE = 2
FLAG_BAD_OFFSETS = 4
FLAG_X_NONPOS = 8


@dataclass
class Params:
    """Hyper-parameters.  Defaults: gamma=0.65 and C=3 (Sec. 5.1); eps is not
    given by the paper, 0.2 is the usual GRPO value."""

    gamma: float = 0.65
    C: float = 3.0
    clip_eps: float = 0.2
    adv_eps: float = 1e-6
    kappa: float = 1.0          # |alpha| of the continuous-reduction ablation (Sec. 5.5)
    x_ema: float = 0.0          # moving-average X (Limitations); 0 keeps X frozen
    entropy_coeff: float = 0.0  # entropy bonus beta (App. A actor.entropy_coeff)
    mode: int = MODE_ACRL
    y_gran: int = Y_GROUP
    agg: int = AGG_SEQ_MEAN_TOKEN_MEAN
    adv_ddof: int = 1
    singleton_rule: int = SINGLETON_MEAN0_STD1
    calib_steps: int = 1
    X_init: float = 0.0


@dataclass
class ControllerState:
    """The controller's whole state: the reference X and its calibration sums
    (Sec. 4.1: X is built before training and then kept fixed)."""

    X: float = 0.0
    calib_sum: float = 0.0
    calib_count: int = 0
    calib_done_steps: int = 0
    step: int = 0
    calibrated: bool = False
    flags: int = 0


def controller_init(params: Params) -> ControllerState:
    """A given X (> 0) skips calibration, as with the printed X values of
    Sec. 5.1; otherwise X is measured on the first batches."""
    st = ControllerState()
    if params.X_init > 0:
        st.X = float(params.X_init)
        st.calibrated = True
    return st


# --------------------------------------------------------------------------
# bf16 handling
# --------------------------------------------------------------------------

def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Widen raw bf16 bit patterns (uint16) to float64 exactly: a bf16 value is
    the upper half of the float32 with the same bits."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return u.view(np.float32).astype(np.float64)


def round_bf16(x) -> np.ndarray:
    """Round float64 values to the nearest bf16 value, ties to even (8
    significant bits), returned as float64.  Written from the format's
    definition: x = f 2^e with f in [0.5, 1); keep f to 8 bits with
    round-half-even.  Finite normal range only (logits)."""
    x = np.asarray(x, dtype=np.float64)
    f, e = np.frexp(x)
    return np.ldexp(np.rint(f * 256.0) / 256.0, e)


def lmhead_logits(hidden, weight) -> np.ndarray:
    """The policy's logits z = H W^T of an LM-head projection, with the
    products summed exactly enough in float64 and the result stored in bf16
    (the training engine's bf16 logits).  hidden [R, K], weight [N, K]."""
    H = np.asarray(hidden, dtype=np.float64)
    Wt = np.asarray(weight, dtype=np.float64)
    return round_bf16(H @ Wt.T)


# --------------------------------------------------------------------------
# a1: log-softmax, sampled-token log-prob, entropy
# --------------------------------------------------------------------------

def token_stats(z: np.ndarray, ids: np.ndarray, mask: np.ndarray | None):
    """Per row t: lse_t = log sum_j exp(z_tj); logp_t = z_{t,a_t} - lse_t is
    log pi(a_t | q, a_<t) as used in r (Eq. grpo_objective), rho (Eq. TIS) and
    d (Eq. distance_metric); H_t = -sum_j p_tj log p_tj is the token entropy
    the paper tracks during training (Sec. 5.1 figures).

    z: float64 [T, V].  Returns (lse, logp, H, flags)."""
    z = np.asarray(z, dtype=np.float64)
    T, V = z.shape
    ids = np.asarray(ids).astype(np.int64)
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    lse = np.zeros(T)
    logp = np.zeros(T)
    H = np.zeros(T)
    flags = 0
    for t in range(T):
        if not m[t]:
            continue
        row = z[t]
        if not np.all(np.isfinite(row)):
            lse[t] = logp[t] = H[t] = np.nan
            flags |= FLAG_NONFINITE
            continue
        zmax = row.max()
        lse[t] = zmax + np.log(np.sum(np.exp(row - zmax)))
        logq = row - lse[t]                 # log-softmax of the row
        p = np.exp(logq)
        H[t] = -np.sum(p * logq)
        a = ids[t]
        if 0 <= a < V:
            logp[t] = logq[a]
        else:
            logp[t] = 0.0
            flags |= FLAG_BAD_ID
    return lse, logp, H, flags


def token_stats_bruteforce(z, ids, mask=None):
    """The same quantities with plain Python loops and math.fsum; only for
    small V (a pin for `token_stats`)."""
    T = len(z)
    out_lse, out_logp, out_H = [], [], []
    for t in range(T):
        if mask is not None and not mask[t]:
            out_lse.append(0.0)
            out_logp.append(0.0)
            out_H.append(0.0)
            continue
        row = [float(v) for v in z[t]]
        big = max(row)
        s = math.fsum(math.exp(v - big) for v in row)
        lse = big + math.log(s)
        probs = [math.exp(v - lse) for v in row]
        ent = -math.fsum(p * math.log(p) for p in probs if p > 0.0)
        out_lse.append(lse)
        out_logp.append(math.log(probs[int(ids[t])]))
        out_H.append(ent)
    return np.array(out_lse), np.array(out_logp), np.array(out_H)


# --------------------------------------------------------------------------
# a2/a3: log-ratio, distance, masked segmented aggregates
# --------------------------------------------------------------------------

def _check_offsets(seq_offsets, group_offsets, T):
    so = np.asarray(seq_offsets, dtype=np.int64)
    go = np.asarray(group_offsets, dtype=np.int64)
    S = len(so) - 1
    ok = (len(so) >= 1 and so[0] == 0 and so[-1] == T and np.all(np.diff(so) >= 0)
          and len(go) >= 1 and go[0] == 0 and go[-1] == S and np.all(np.diff(go) >= 0))
    return so, go, bool(ok)


def seq_discrepancy(logp_pi, logp_mu, mask, seq_offsets, group_offsets, entropy=None):
    """Per token: lr_t = log pi_old(a_t) - log mu(a_t) (the log of rho in
    Eq. TIS) and d_t = |pi_old(a_t) - mu(a_t)| (Eq. distance_metric).
    Per sequence i: n_i = |a_i| (valid tokens), D_i = (1/n_i) sum_t d_t, the
    MIS log-ratio S_i = sum_t lr_t = log rho_i (Eq. MIS), max/sum/sum-of-squares
    of d and the mean entropy.  Per group g: G_g valid sequences and
    Y_g = (1/G_g) sum_i D_i (the current discrepancy Y defined after Eq. ACRL).
    Batch: token mean/max/std of d (the curves of Sec. 5.1), the prompt mean of
    Y_g (the step discrepancy of the X-evolution table), token-mean entropy and
    log-ratio.

    Returns (lr, d, seq, grp, batch, flags) with seq/grp/batch dicts."""
    pi = np.asarray(logp_pi, dtype=np.float64)
    mu = np.asarray(logp_mu, dtype=np.float64)
    T = len(pi)
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    so, go, ok = _check_offsets(seq_offsets, group_offsets, T)
    flags = 0 if ok else FLAG_BAD_OFFSETS
    S, Gn = len(so) - 1, len(go) - 1

    with np.errstate(invalid="ignore"):
        lr = np.where(m, pi - mu, 0.0)
    d = np.where(m, np.abs(np.exp(pi) - np.exp(mu)), 0.0)
    if np.any(np.isnan(lr[m])):
        flags |= FLAG_NONFINITE         # a NaN log-prob on either side of a valid token
    Hm = None if entropy is None else np.where(m, np.asarray(entropy, dtype=np.float64), 0.0)

    seq = {k: np.zeros(S) for k in ("mean_d", "max_d", "sum_d", "sum_d2", "sum_lr", "mean_H")}
    seq["n"] = np.zeros(S, dtype=np.int64)
    seq["group"] = np.full(S, -1, dtype=np.int64)
    for g in range(Gn):
        seq["group"][go[g]:go[g + 1]] = g
    for i in range(S):
        sl = slice(so[i], so[i + 1])
        mi = m[sl]
        n = int(mi.sum())
        seq["n"][i] = n
        if n == 0:
            continue
        di = d[sl][mi]
        seq["sum_d"][i] = di.sum()
        seq["sum_d2"][i] = (di * di).sum()
        seq["max_d"][i] = di.max()
        seq["mean_d"][i] = di.sum() / n
        seq["sum_lr"][i] = lr[sl][mi].sum()
        if Hm is not None:
            seq["mean_H"][i] = Hm[sl][mi].sum() / n

    grp = {"n_valid_seqs": np.zeros(Gn, dtype=np.int64), "n_tokens": np.zeros(Gn, dtype=np.int64),
           "Y": np.zeros(Gn)}
    for g in range(Gn):
        members = range(go[g], go[g + 1])
        valid = [i for i in members if seq["n"][i] > 0]
        grp["n_valid_seqs"][g] = len(valid)
        grp["n_tokens"][g] = sum(int(seq["n"][i]) for i in members)
        if valid:
            grp["Y"][g] = sum(seq["mean_d"][i] for i in valid) / len(valid)

    valid_g = grp["n_valid_seqs"] > 0
    N = int(m.sum())
    dv = d[m]
    batch = {
        "n_tokens": N,
        "n_groups_valid": int(valid_g.sum()),
        "n_seqs_valid": int((seq["n"] > 0).sum()),
        "d_mean": float(dv.mean()) if N else 0.0,
        "d_max": float(dv.max()) if N else 0.0,
        "d_std": float(dv.std()) if N else 0.0,
        "Y_sum": float(grp["Y"][valid_g].sum()),
        "Y_mean": float(grp["Y"][valid_g].mean()) if valid_g.any() else 0.0,
        "H_mean": float(Hm[m].mean()) if (Hm is not None and N) else 0.0,
        "lr_mean": float(lr[m].mean()) if N else 0.0,
    }
    return lr, d, seq, grp, batch, flags


# --------------------------------------------------------------------------
# a4: GRPO advantage
# --------------------------------------------------------------------------

def grpo_advantage(rewards, group_offsets, params: Params):
    """A_i = (R_i - mean_g R) / std_g R over the responses of one prompt
    (Sec. 2, the definition under Eq. grpo_objective), with std taken with
    `adv_ddof` degrees of freedom and `adv_eps` added to it."""
    R = np.asarray(rewards, dtype=np.float64)
    go = np.asarray(group_offsets, dtype=np.int64)
    A = np.zeros(len(R))
    for g in range(len(go) - 1):
        r = R[go[g]:go[g + 1]]
        G = len(r)
        if G == 0:
            continue
        if G == 1:
            A[go[g]] = r[0] if params.singleton_rule == SINGLETON_MEAN0_STD1 else 0.0
            continue
        if np.all(r == r[0]):
            # equal rewards: every R_i - mean is exactly 0, so A = 0 (0/0 read as 0 when adv_eps = 0); decided
            # here exactly, since a float64 mean of values with full 53-bit significands can miss them by an ulp
            continue
        mean = r.sum() / G
        var = ((r - mean) ** 2).sum() / (G - params.adv_ddof) if G > params.adv_ddof else 0.0
        den = math.sqrt(var) + params.adv_eps
        A[go[g]:go[g + 1]] = (r - mean) / den if den > 0 else 0.0
    return A


# --------------------------------------------------------------------------
# a5: controller step and importance weights
# --------------------------------------------------------------------------

def controller_step(state: ControllerState, params: Params, lr, mask, seq_offsets, group_offsets,
                    seq, grp, batch, adv):
    """Calibrate or apply the reference X (Sec. 4.1), then the per-sequence
    exponent alpha_i = gamma * sign(A_i) * (1 - Y/X) (Sec. 4.1, after
    Eq. ACRL) and per-token weights:
      ACRL: min(rho_t, C) with rho_t = (pi_old/mu)^alpha_i   (Eq. ACRL)
      TIS : min(pi_old/mu, C)                                (Eq. TIS)
      MIS : rho_i * 1{rho_i <= C}, rho_i = prod_t pi_old/mu   (Eq. MIS)
      NONE: 1                                                (Eq. grpo_objective)
    Returns (weight [T], alpha [S], new_state, info dict, flags).  `state` is
    not modified."""
    st = ControllerState(**vars(state))
    lr = np.asarray(lr, dtype=np.float64)
    T = len(lr)
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    so = np.asarray(seq_offsets, dtype=np.int64)
    S = len(so) - 1
    A = np.asarray(adv, dtype=np.float64)
    flags = 0

    applying = True
    was_calibrated = st.calibrated
    if not st.calibrated:
        st.calib_sum += batch["Y_sum"]
        st.calib_count += batch["n_groups_valid"]
        st.calib_done_steps += 1
        if st.calib_done_steps >= params.calib_steps:
            st.X = st.calib_sum / st.calib_count if st.calib_count > 0 else 0.0
            st.calibrated = True
        else:
            applying = False
    st.step += 1

    X = st.X
    if params.mode in (MODE_ACRL, MODE_ACRL_FALLBACK) and applying and not X > 0:
        flags |= FLAG_X_NONPOS
    # Moving-average X (Limitations): this step uses X, later steps the update.
    if was_calibrated and params.x_ema > 0:
        st.X = (1.0 - params.x_ema) * X + params.x_ema * batch["Y_mean"]

    logC = math.log(params.C)
    alpha = np.zeros(S)
    w = np.zeros(T)
    n_trunc = 0
    for i in range(S):
        n_i = int(seq["n"][i])
        if params.mode == MODE_TIS or params.mode == MODE_MIS:
            alpha[i] = 1.0
        elif params.mode == MODE_ACRL_CONTINUOUS and n_i > 0:
            # Sec. 5.5: alpha = -1 (or -3) where A > 0, +1 (or +3) where A < 0
            alpha[i] = -params.kappa * np.sign(A[i])
        elif params.mode in (MODE_ACRL, MODE_ACRL_FALLBACK) and applying and X > 0 and n_i > 0:
            if params.y_gran == Y_GROUP:
                Y = grp["Y"][seq["group"][i]]
            elif params.y_gran == Y_SEQUENCE:
                Y = seq["mean_d"][i]
            else:
                Y = batch["Y_mean"]
            alpha[i] = params.gamma * np.sign(A[i]) * (1.0 - Y / X)
            if params.mode == MODE_ACRL_FALLBACK and not Y > X:
                alpha[i] = 0.0      # Sec. 5.5: plain GRPO update when Y < X
        for t in range(so[i], so[i + 1]):
            if not m[t]:
                continue
            if params.mode == MODE_NONE:
                w[t] = 1.0
            elif params.mode == MODE_MIS:
                S_i = seq["sum_lr"][i]
                w[t] = math.exp(S_i) if S_i <= logC else 0.0     # a NaN S_i fails the test: weight 0
                n_trunc += S_i > logC
            else:
                # rho^0 = 1 even where the log-ratio is infinite (mu = 0); a NaN log-ratio gets weight 0
                log_rho = 0.0 if alpha[i] == 0.0 else alpha[i] * lr[t]
                w[t] = 0.0 if math.isnan(log_rho) else math.exp(min(log_rho, logC))
                n_trunc += log_rho > logC
    N = int(m.sum())
    valid_seq = np.asarray(seq["n"]) > 0
    info = {
        "X": X,
        "trunc_frac": n_trunc / N if N else 0.0,
        "w_mean": float(w[m].mean()) if N else 0.0,
        "alpha_mean": float(alpha[valid_seq].mean()) if valid_seq.any() else 0.0,
    }
    st.flags |= flags
    return w, alpha, st, info, flags


# --------------------------------------------------------------------------
# a6: policy loss and its gradient with respect to the logits
# --------------------------------------------------------------------------

def _seq_of_rows(so, T):
    owner = np.full(T, -1, dtype=np.int64)
    for i in range(len(so) - 1):
        owner[so[i]:so[i + 1]] = i
    return owner


def loss_grad_logits(z, ids, mask, lse, old_logp, adv, weight, seq_offsets, seq, grp, batch,
                     params: Params, rows=None):
    """Loss of Eq. ACRL (Eq. TIS / Eq. MIS / Eq. grpo_objective for the other
    modes: the weight is the only difference) and its gradient w.r.t. the
    logits.  Per valid token, with r_t = exp(logp_t - old_logp_t) (r = 1 when
    `old_logp` is None, the one-update-per-rollout setting of App. A):
        loss_t = -w_t * min(r_t A_i, clip(r_t, 1-eps, 1+eps) A_i) / norm_t
    with norm_t = Q_eff * G_g * n_i (the 1/G sum_i 1/|a_i| sum_t of the
    objective, averaged over prompts) or the valid-token count (TOKEN_MEAN).
    The weight w_t is a constant (it is built from theta_old).  By the chain
    rule, d logp_t / d z_tj = 1[j = a_t] - p_tj and dr/dz = r dlogp/dz, so
        dL/dz_tj = coef_t (p_tj - 1[j = a_t]),
        coef_t = w_t g_t r_t A_i / norm_t,
    where g_t = 1 when the unclipped branch is the minimum (A >= 0 and
    r <= 1+eps, or A < 0 and r >= 1-eps) and 0 otherwise.

    z: float64 [T, V] (or only the rows listed in `rows`, in that order).
    lse: None to recompute from z.  Returns (grad [len(rows), V],
    token_loss [T] (NaN where not computed), loss over the computed rows)."""
    z = np.asarray(z, dtype=np.float64)
    so = np.asarray(seq_offsets, dtype=np.int64)
    T = len(np.asarray(weight))
    rows = np.arange(T) if rows is None else np.asarray(rows, dtype=np.int64)
    V = z.shape[1]
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    ids = np.asarray(ids).astype(np.int64)
    A = np.asarray(adv, dtype=np.float64)
    w = np.asarray(weight, dtype=np.float64)
    owner = _seq_of_rows(so, T)
    eps = params.clip_eps
    grad = np.zeros((len(rows), V))
    token_loss = np.full(T, np.nan)
    total = []
    for k, t in enumerate(rows):
        i = owner[t]
        a = ids[t]
        if i < 0 or not m[t] or not (0 <= a < V):
            token_loss[t] = 0.0
            total.append(0.0)
            continue
        g_idx = int(seq["group"][i])
        if params.agg == AGG_TOKEN_MEAN:
            norm = float(batch["n_tokens"])
        else:
            norm = float(batch["n_groups_valid"]) * float(grp["n_valid_seqs"][g_idx]) * float(seq["n"][i])
        Ai = A[i]
        beta = params.entropy_coeff / norm
        if w[t] * Ai == 0.0 and beta == 0.0:
            # reading c18: a row whose weighted advantage is 0 contributes nothing; its logits are not needed
            token_loss[t] = 0.0
            total.append(0.0)
            continue
        row = z[k]
        with np.errstate(invalid="ignore"):     # a non-finite row gives a non-finite lse, handled below
            if lse is None:
                top = row.max()
                lse_t = top + np.log(np.sum(np.exp(row - top)))
            else:
                lse_t = float(lse[t])
            logp_t = row[a] - lse_t
        old_t = math.nan if old_logp is None else float(old_logp[t])
        if not (math.isfinite(lse_t) and math.isfinite(logp_t)) or (old_logp is not None and math.isnan(old_t)):
            # reading c17: a row whose log-sum-exp or log-prob is not finite (a NaN or an infinity among its
            # logits), or whose old log-prob is NaN, has no defined surrogate: NaN token loss and gradient row
            token_loss[t] = math.nan
            grad[k] = math.nan
            total.append(math.nan)
            continue
        r = 1.0 if old_logp is None else math.exp(logp_t - old_t)
        rc = min(max(r, 1.0 - eps), 1.0 + eps)
        surrogate = min(r * Ai, rc * Ai)
        token_loss[t] = -w[t] * surrogate / norm
        gate = (Ai >= 0 and r <= 1.0 + eps) or (Ai < 0 and r >= 1.0 - eps)
        coef = w[t] * (1.0 if gate else 0.0) * r * Ai / norm
        if coef == 0.0 and beta == 0.0:
            total.append(token_loss[t])
            continue
        logq = row - lse_t
        p = np.exp(logq)
        g = coef * p
        g[a] -= coef
        if beta != 0.0:
            # entropy bonus -beta H_t / norm_t; dH/dz_j = -p_j (log p_j + H)
            H_t = -np.sum(p * logq)
            token_loss[t] -= beta * H_t
            g += beta * p * (logq + H_t)
        total.append(token_loss[t])
        grad[k] = g
    return grad, token_loss, math.fsum(total)


def _norms(mask, seq_offsets, seq, grp, batch, params: Params):
    """norm_t of the aggregation: Q_eff * G_g * n_i (the prompt average of
    (1/G) sum_i (1/|a_i|) sum_t in Eq. grpo_objective) or the token count."""
    so = np.asarray(seq_offsets, dtype=np.int64)
    T = int(so[-1])
    owner = _seq_of_rows(so, T)
    norm = np.zeros(T)
    for t in range(T):
        i = owner[t]
        if i < 0:
            continue
        if params.agg == AGG_TOKEN_MEAN:
            norm[t] = float(batch["n_tokens"])
        else:
            g = int(seq["group"][i])
            norm[t] = float(batch["n_groups_valid"]) * float(grp["n_valid_seqs"][g]) * float(seq["n"][i])
    return owner, norm


def loss_coefficients(weight, adv, mask, seq_offsets, seq, grp, batch, params: Params):
    """Per-token factor w_t A_i / norm_t that multiplies grad r_t in Eq. ACRL
    (0 on masked tokens)."""
    w = np.asarray(weight, dtype=np.float64)
    A = np.asarray(adv, dtype=np.float64)
    T = len(w)
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    owner, norm = _norms(mask, seq_offsets, seq, grp, batch, params)
    coef = np.zeros(T)
    for t in range(T):
        if m[t] and owner[t] >= 0 and norm[t] > 0:
            coef[t] = w[t] * A[owner[t]] / norm[t]
    return coef


def entropy_coefficients(mask, seq_offsets, seq, grp, batch, params: Params):
    """Per-token factor beta / norm_t of the entropy bonus (0 on masked tokens)."""
    so = np.asarray(seq_offsets, dtype=np.int64)
    T = int(so[-1])
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    owner, norm = _norms(mask, seq_offsets, seq, grp, batch, params)
    out = np.zeros(T)
    ok = m & (owner >= 0) & (norm > 0)
    out[ok] = params.entropy_coeff / norm[ok]
    return out


def surrogate_loss(logp, old_logp, adv, weight, mask, seq_offsets, seq, grp, batch, params: Params, entropy=None):
    """Token losses -w_t min(r A, clip(r) A) / norm_t of Eq. ACRL from the
    current log-probs alone (r = exp(logp - old_logp), or 1 without old_logp),
    minus beta H_t / norm_t when an entropy bonus and the entropies are given.
    Returns (token_loss [T], total)."""
    w = np.asarray(weight, dtype=np.float64)
    A = np.asarray(adv, dtype=np.float64)
    T = len(w)
    m = np.ones(T, dtype=bool) if mask is None else (np.asarray(mask) != 0)
    owner, norm = _norms(mask, seq_offsets, seq, grp, batch, params)
    eps = params.clip_eps
    tl = np.zeros(T)
    for t in range(T):
        i = owner[t]
        if not m[t] or i < 0 or norm[t] <= 0:
            continue
        r = 1.0 if old_logp is None else math.exp(float(logp[t]) - float(old_logp[t]))
        rc = min(max(r, 1.0 - eps), 1.0 + eps)
        tl[t] = -w[t] * min(r * A[i], rc * A[i]) / norm[t]
        if entropy is not None and params.entropy_coeff:
            tl[t] -= params.entropy_coeff * float(entropy[t]) / norm[t]
    return tl, math.fsum(tl)


# --------------------------------------------------------------------------
# whole step (for tests and the CPU baseline)
# --------------------------------------------------------------------------

@dataclass
class StepResult:
    lse: np.ndarray
    logp: np.ndarray
    H: np.ndarray
    lr: np.ndarray
    d: np.ndarray
    seq: dict
    grp: dict
    batch: dict
    adv: np.ndarray
    weight: np.ndarray
    alpha: np.ndarray
    state: ControllerState
    info: dict
    grad: np.ndarray
    token_loss: np.ndarray
    loss: float
    flags: int = 0
    extra: dict = field(default_factory=dict)


def step(z, ids, mask, logp_mu, rewards, seq_offsets, group_offsets, params: Params,
         state: ControllerState | None = None):
    """One on-policy pass in the paper's order: log-probs and entropy of pi,
    discrepancy statistics against mu, GRPO advantages, the controller, then
    the loss gradient with respect to the logits (theta = theta_old, r = 1)."""
    if state is None:
        state = controller_init(params)
    lse, logp, H, f1 = token_stats(z, ids, mask)
    lr, d, seq, grp, batch, f2 = seq_discrepancy(logp, logp_mu, mask, seq_offsets, group_offsets, H)
    adv = grpo_advantage(rewards, group_offsets, params)
    w, alpha, st, info, f3 = controller_step(state, params, lr, mask, seq_offsets, group_offsets,
                                             seq, grp, batch, adv)
    grad, tl, loss = loss_grad_logits(z, ids, mask, lse, None, adv, w, seq_offsets, seq, grp, batch,
                                      params)
    return StepResult(lse, logp, H, lr, d, seq, grp, batch, adv, w, alpha, st, info, grad, tl, loss,
                      f1 | f2 | f3)
