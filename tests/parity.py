"""Helpers for comparing the CUDA path (through the C ABI) with the float64
oracle on the same seeded inputs.  Tolerances are the ones the method's
arithmetic supports (bf16 in, fp32 accumulation):
  * log-probs / lse: 2e-4 absolute; a per-token probability distance d
    compared with the fp64 chain inherits that bar as |dd| <= pi * 2e-4, and
    is checked tightly (1e-3 relative) when the oracle is fed the GPU's own
    fp32 log-probs;
  * entropy, weights, alpha, aggregates, X, batch statistics, loss: 1e-3
    relative (entropy with a 1e-5 absolute floor; the scalar loss with a floor
    of 1e-6 * sum |token loss|, since the token losses can cancel);
  * bf16 gradient elements: 1e-2 relative; an element whose reference is
    below 2^-125 may come back as 0 (the exp2 flushes subnormals); the
    sampled column, coef * (p_a - 1), carries the fp32 error of logp_a, so it
    also gets an absolute floor of 1e-5 * |coef|.
Integer outputs (counts, group indices, flags) must match exactly."""

from __future__ import annotations

import atexit
import concurrent.futures
import multiprocessing
import os

import numpy as np

import oracle as O

TOL_LOGP = 2e-4
TOL_REL = 1e-3
TOL_GRAD = 1e-2
FTZ = 2.0 ** -125


def host(t):
    return t.detach().cpu().numpy()


def oracle_params(p) -> O.Params:
    return O.Params(gamma=float(p.gamma), C=float(p.C), clip_eps=float(p.clip_eps), adv_eps=float(p.adv_eps),
                    kappa=float(p.kappa), x_ema=float(p.x_ema), entropy_coeff=float(p.entropy_coeff),
                    mode=int(p.mode), y_gran=int(p.y_gran), agg=int(p.agg), adv_ddof=int(p.adv_ddof),
                    singleton_rule=int(p.singleton_rule), calib_steps=int(p.calib_steps), X_init=float(p.X_init))


def rows_bits(t, rows, V: int) -> np.ndarray:
    """The raw bf16 bits (uint16) of `rows` of a [T, ld] tensor, first V columns."""
    import torch
    idx = torch.as_tensor(np.asarray(rows, dtype=np.int64), device=t.device)
    return t.index_select(0, idx)[:, :V].contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def rows_f64(logits, rows, V: int) -> np.ndarray:
    """Exact float64 copy of the bf16 logits of `rows` (first V columns)."""
    return O.bf16_bits_to_f64(rows_bits(logits, rows, V))


def grad_rows(grad, rows, V: int) -> np.ndarray:
    import torch
    idx = torch.as_tensor(np.asarray(rows, dtype=np.int64), device=grad.device)
    return grad.index_select(0, idx)[:, :V].float().cpu().numpy().astype(np.float64)


def assert_close_rel(got, ref, rel=TOL_REL, floor=0.0, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    bad = ~(np.abs(got - ref) <= rel * np.abs(ref) + floor)   # a NaN on one side only is a mismatch
    bad &= ~(np.isnan(got) & np.isnan(ref)) & (got != ref)    # NaN against NaN, or equal infinities, match
    if bad.any():
        k = np.flatnonzero(bad.ravel())[:5]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside rel {rel} floor {floor}; "
                             f"got {got.ravel()[k]} ref {ref.ravel()[k]} at {k}")


def assert_close_abs(got, ref, tol, what=""):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    bad = ~(np.abs(got - ref) <= tol)   # a NaN on one side only is a mismatch
    bad &= ~(np.isnan(got) & np.isnan(ref)) & (got != ref)    # NaN against NaN, or equal infinities, match
    if bad.any():
        k = np.flatnonzero(bad.ravel())[:5]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside abs {tol}; got {got.ravel()[k]} "
                             f"ref {ref.ravel()[k]} at {k}")


def assert_grad_rows(got, ref, coef_eff, ids_rows, what="grad", row_floor=0.0):
    """got/ref [R, V]; coef_eff [R] = the reference coef_t g_t r_t.  With an
    entropy bonus an element is p_j (c + e (z_j - lse + H)), whose bracket can
    cancel; `row_floor` then adds row_floor * max_j |ref[t, j]| per row."""
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    tol = TOL_GRAD * np.abs(ref)
    tol = np.maximum(tol, np.where(np.abs(ref) < FTZ, FTZ, 0.0))
    if row_floor:
        tol += row_floor * np.abs(ref).max(axis=1, keepdims=True)
    R = ref.shape[0]
    cols = np.asarray(ids_rows, dtype=np.int64)
    ok_ids = (cols >= 0) & (cols < ref.shape[1])
    r_idx = np.arange(R)[ok_ids]
    tol[r_idx, cols[ok_ids]] += 1e-5 * np.abs(np.asarray(coef_eff)[ok_ids])
    # a NaN on one side only is a mismatch; NaN against NaN, or equal infinities, match
    bad = ~(np.abs(got - ref) <= tol) & ~(np.isnan(got) & np.isnan(ref)) & (got != ref)
    if bad.any():
        rr, cc = np.nonzero(bad)
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} elements off; first rows {rr[:5]} cols {cc[:5]} "
                             f"got {got[rr[:5], cc[:5]]} ref {ref[rr[:5], cc[:5]]}")


def compare_seq(gpu_seq, ref_seq, what="seq"):
    assert np.array_equal(gpu_seq["n"], ref_seq["n"]), f"{what}.n"
    assert np.array_equal(gpu_seq["group"], ref_seq["group"]), f"{what}.group"
    assert_close_rel(gpu_seq["mean_d"], ref_seq["mean_d"], floor=1e-7, what=f"{what}.mean_d")
    assert_close_rel(gpu_seq["max_d"], ref_seq["max_d"], floor=1e-7, what=f"{what}.max_d")
    assert_close_rel(gpu_seq["sum_d"], ref_seq["sum_d"], floor=1e-6, what=f"{what}.sum_d")
    assert_close_rel(gpu_seq["sum_d2"], ref_seq["sum_d2"], floor=1e-7, what=f"{what}.sum_d2")
    # S_i = log rho_i: an absolute quantity; its exp is the MIS weight
    assert_close_abs(gpu_seq["sum_lr"], ref_seq["sum_lr"], TOL_REL * np.maximum(1.0, np.abs(ref_seq["sum_lr"])),
                     what=f"{what}.sum_lr")


def compare_grp(gpu_grp, ref_grp, what="grp"):
    assert np.array_equal(gpu_grp["n_valid_seqs"], ref_grp["n_valid_seqs"]), f"{what}.n_valid_seqs"
    assert np.array_equal(gpu_grp["n_tokens"], ref_grp["n_tokens"]), f"{what}.n_tokens"
    assert_close_rel(gpu_grp["Y"], ref_grp["Y"], floor=1e-9, what=f"{what}.Y")


def compare_batch(gb, rb, what="batch"):
    assert int(gb["n_tokens"]) == rb["n_tokens"], f"{what}.n_tokens"
    assert int(gb["n_groups_valid"]) == rb["n_groups_valid"], f"{what}.n_groups_valid"
    assert int(gb["n_seqs_valid"]) == rb["n_seqs_valid"], f"{what}.n_seqs_valid"
    for k in ("d_mean", "d_max", "d_std", "Y_sum", "Y_mean"):
        assert_close_rel(gb[k], rb[k], floor=1e-9, what=f"{what}.{k}")
    assert_close_rel(gb["H_mean"], rb["H_mean"], floor=1e-5, what=f"{what}.H_mean")
    assert_close_abs(gb["lr_mean"], rb["lr_mean"], TOL_LOGP, what=f"{what}.lr_mean")


def assert_loss(got, ref, ref_token_loss, what="loss"):
    """Scalar loss: 1e-3 relative, with a floor of 1e-6 * sum |token loss| for
    batches whose token losses cancel (e.g. every weight 1: sum_i A_i = 0)."""
    floor = 1e-6 * float(np.nansum(np.abs(np.asarray(ref_token_loss, dtype=np.float64)))) + 1e-30
    assert_close_rel(got, ref, floor=floor, what=what)


# --------------------------------------------------------------------------
# the vocabulary-wide outputs of many rows, checked in parallel
# --------------------------------------------------------------------------

_POOL = None


def oracle_pool():
    """Worker processes for the oracle's per-row work, one per host core (at
    most 16).  Spawned, so that none inherits this process's CUDA context;
    they import numpy and the oracle only."""
    global _POOL
    if _POOL is None:
        n = max(1, min(16, len(os.sched_getaffinity(0))))
        _POOL = (concurrent.futures.ProcessPoolExecutor(max_workers=n,
                                                        mp_context=multiprocessing.get_context("spawn")), n)
        atexit.register(_POOL[0].shutdown)
    return _POOL


def _vocab_rows_block(zbits, gbits, rr, T, ids_r, mask_r, w_r, coef_r, adv, so, seq, grp, batch, op, lse_g, logp_g,
                      ent_g):
    """One block of rows in a worker: the oracle's log-softmax of the exact
    float64 logits against the GPU's lse / logp / entropy, then the oracle's
    gradient rows (Eq. ACRL) against the GPU's bf16 gradient rows.  Returns
    (rows, oracle logp, oracle entropy)."""
    z = O.bf16_bits_to_f64(zbits)
    olse, ologp, oH, f = O.token_stats(z, ids_r, mask_r)
    assert f == 0, f"oracle flags {f}"
    assert_close_abs(lse_g, olse, TOL_LOGP, "lse")
    assert_close_abs(logp_g, ologp, TOL_LOGP, "logp")
    assert_close_rel(ent_g, oH, floor=1e-5, what="entropy")
    if gbits is not None:
        full = np.zeros(T)
        full[rr] = olse
        ids_full = np.zeros(T, dtype=np.int64)
        ids_full[rr] = ids_r
        mask_full = np.zeros(T, dtype=np.uint8)
        mask_full[rr] = mask_r
        w_full = np.zeros(T)
        w_full[rr] = w_r
        ograd, _, _ = O.loss_grad_logits(z, ids_full, mask_full, full, None, adv, w_full, so, seq, grp, batch, op,
                                         rows=rr)
        assert_grad_rows(O.bf16_bits_to_f64(gbits), ograd, coef_r, ids_r)
    return rr, ologp, oH


class VocabRowCheck:
    """Element-by-element check of the vocabulary-wide outputs (a1: lse, logp,
    entropy; a6: the gradient rows) of sampled rows against the oracle's own
    float64 log-softmax and gradient, in blocks of rows spread over the
    oracle pool.  `ref` holds the O(T) references the gradient needs (adv, w,
    coef, seq, grp, batch).  The oracle's logp and entropy of every checked
    row are kept (`oracle_logp`, `oracle_entropy`) for the oracle's own chain
    on whole responses."""

    def __init__(self, T, ids, mask, seq_offsets, ref, op, block=256):
        self.pool, self.n = oracle_pool()
        self.T, self.ids, self.mask = T, np.asarray(ids), np.asarray(mask)
        self.so = np.asarray(seq_offsets)
        self.ref, self.op, self.block = ref, op, block
        self.pending = set()
        self.oracle_logp, self.oracle_entropy = {}, {}
        self.rows_checked = 0

    def _collect(self, futures):
        for f in futures:
            rr, lp, H = f.result()      # re-raises a worker's AssertionError here
            self.oracle_logp.update(zip(rr.tolist(), lp.tolist()))
            self.oracle_entropy.update(zip(rr.tolist(), H.tolist()))
            self.rows_checked += len(rr)

    def submit(self, logits, V, rows, lse, logp, entropy, grad=None, grad_row0=0):
        """Queue `rows` (global row indices) for checking.  `grad` holds the
        gradient rows from global row `grad_row0` on (a chunk buffer), or is
        None to check the statistics alone.  The rows' data are copied to the
        host before this returns, so the buffers may be reused."""
        rows = np.asarray(rows, dtype=np.int64)
        lse_h, logp_h, ent_h = host(lse), host(logp), host(entropy)
        r = self.ref
        for k in range(0, len(rows), self.block):
            rr = rows[k:k + self.block]
            zb = rows_bits(logits, rr, V)
            gb = None if grad is None else rows_bits(grad, rr - grad_row0, V)
            while len(self.pending) >= 2 * self.n:
                done, self.pending = concurrent.futures.wait(self.pending,
                                                             return_when=concurrent.futures.FIRST_COMPLETED)
                self._collect(done)
            self.pending.add(self.pool.submit(
                _vocab_rows_block, zb, gb, rr, self.T, self.ids[rr], self.mask[rr], r["w"][rr], r["coef"][rr],
                r["adv"], self.so, r["seq"], r["grp"], r["batch"], self.op, lse_h[rr], logp_h[rr], ent_h[rr]))

    def finish(self):
        """Wait for every queued block; returns the number of rows checked."""
        done, _ = concurrent.futures.wait(self.pending)
        self.pending = set()
        self._collect(done)
        return self.rows_checked
