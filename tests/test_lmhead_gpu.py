"""The fused LM-head path (tcgen05 GEMM with the log-softmax statistics in
its epilogue, then the merge) against the float64 oracle: logits within one
bf16 ulp of the exactly rounded product, lse/logp/entropy within the bars of
the statistics pass, and the whole ACRL chain on the workload of 32,768
tokens x 4,096 hidden x 151,936 vocabulary on sampled rows."""

import numpy as np
import pytest
import torch

import oracle as O
import workloads as W
from parity import (TOL_LOGP, assert_close_abs, assert_close_rel, assert_grad_rows, assert_loss, compare_batch,
                    compare_seq, grad_rows, host, oracle_params, rows_f64)

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import _abi, api  # noqa: E402

DEV = "cuda"


def _f64(t):
    return t.detach().to(torch.float64).cpu().numpy()


def _check_logits(got_bf16, ref, abs_sum, K, what="logits"):
    """The GPU rounds an fp32 sum of K products to bf16, the oracle the exact
    sum: they may differ by one bf16 ulp of the result plus the fp32
    accumulation error, bounded here by 8 sqrt(K) 2^-24 sum_k |h_k w_k| (a
    dropped or repeated K slice would be off by ~ sum / (K/16), far beyond it).
    Almost every element must agree exactly."""
    got = _f64(got_bf16)
    ulp = np.ldexp(1.0, np.frexp(np.abs(ref))[1] - 8)
    tol = ulp * 1.0000001 + 8.0 * np.sqrt(K) * 2.0 ** -24 * abs_sum + 1e-30
    bad = np.abs(got - ref) > tol
    assert not bad.any(), f"{what}: {bad.sum()} of {bad.size} off by more than the bound"
    assert np.mean(got == ref) > 0.99


# also: one row and a vocabulary narrower than a 32-column store block; an odd number of row tiles with a
# ragged K; K narrower than one 64-column slab; 66 row tiles, i.e. three bands of row tiles (32, 32 and a ragged
# 2) with a ragged last tile; one short of / one past the 128-row and 256-column tile edges with K off the
# 64-column slab
@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (200, 1000, 328), (384, 2304, 4096), (130, 151936, 64),
                                   (1, 8, 64), (257, 520, 72), (5, 40, 8), (8322, 1000, 64),
                                   (127, 255, 16), (129, 257, 136), (256, 512, 200), (255, 33, 24)])
def test_lmhead_small_shapes(M, N, K):
    gen = torch.Generator(device=DEV).manual_seed(M * 7 + N + K)
    H = torch.randn((M, K), generator=gen, device=DEV).to(torch.bfloat16)
    Wt = (0.02 * torch.randn((N, K), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, N, (M,), generator=gen, device=DEV, dtype=torch.int32)
    mask = (torch.rand(M, generator=gen, device=DEV) < 0.9).to(torch.uint8)
    flags = api.new_flags()
    logits, partials = api.lmhead_logits_stats(H, Wt, N=N, flags=flags)
    lse, logp, ent = api.lmhead_merge(partials, logits, ids, mask, N=N, flags=flags)
    assert api.read_flags(flags) == 0
    z = O.lmhead_logits(_f64(H), _f64(Wt))
    _check_logits(logits[:, :N], z, np.abs(_f64(H)) @ np.abs(_f64(Wt)).T, K)
    # merge against the statistics of the logits the GEMM stored (the epilogue's own arithmetic) ...
    zg = rows_f64(logits, np.arange(M), N)
    olse, ologp, oH, _ = O.token_stats(zg, host(ids), host(mask))
    assert_close_abs(host(lse), olse, 1e-5 + 1e-6 * np.abs(olse), "lse (stored logits)")
    assert_close_abs(host(logp), ologp, 2e-5, "logp (stored logits)")
    assert_close_rel(host(ent), oH, rel=1e-4, floor=1e-6, what="entropy (stored logits)")
    # ... and against the oracle's own chain.  A logit whose exact value sits within the fp32 accumulation error
    # of a bf16 rounding boundary may be stored one ulp off the oracle's rounding (both roundings are valid,
    # _check_logits allows it); lse moves by sum_j p_j |dz_j| and log p by that plus |dz_a| in such a row.
    olse, ologp, oH, _ = O.token_stats(z, host(ids), host(mask))
    dz = np.abs(zg - z)
    p = np.exp(z - olse[:, None])
    shift = (p * dz).sum(axis=1)
    a = host(ids)
    assert_close_abs(host(lse), olse, TOL_LOGP + shift, "lse")
    assert_close_abs(host(logp), ologp, TOL_LOGP + shift + dz[np.arange(M), a], "logp")
    assert_close_rel(host(ent), oH, floor=1e-5, what="entropy")


def test_lmhead_matches_token_stats_on_same_logits():
    """The fused statistics equal acrl_token_stats run on the logits the GEMM wrote."""
    M, N, K = 256, 32000, 512
    gen = torch.Generator(device=DEV).manual_seed(5)
    H = torch.randn((M, K), generator=gen, device=DEV).to(torch.bfloat16)
    Wt = (0.05 * torch.randn((N, K), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, N, (M,), generator=gen, device=DEV, dtype=torch.int32)
    logits, partials = api.lmhead_logits_stats(H, Wt, N=N)
    lse, logp, ent = api.lmhead_merge(partials, logits, ids, None, N=N)
    lse2, logp2, ent2 = api.token_stats(logits, ids, None, V=N)
    torch.cuda.synchronize()
    assert_close_abs(host(lse), host(lse2), 1e-5, "lse")
    assert_close_abs(host(logp), host(logp2), 1e-5, "logp")
    assert_close_rel(host(ent), host(ent2), rel=1e-5, floor=1e-6, what="entropy")


def test_lmhead_workload_full_chain():
    """32,768 tokens x 4,096 x 151,936: GEMM + merge, discrepancy, advantages,
    controller, gradient on the stored logits; the O(T) stages on every row,
    the vocabulary-wide outputs on 1,024 random rows plus the first and last
    row of every 128-row tile."""
    torch.cuda.empty_cache()
    b = W.generate_lmhead(device=DEV)
    p = acrl.Params()
    op = oracle_params(p)
    flags = api.new_flags()
    logits, partials = api.lmhead_logits_stats(b.hidden, b.weight, N=b.N, flags=flags)
    lse, logp, ent = api.lmhead_merge(partials, logits, b.ids, b.mask, N=b.N, flags=flags)
    del partials
    disc = api.seq_discrepancy(logp, b.logp_mu, b.mask, b.seq_offsets, b.group_offsets, ent, flags=flags)
    adv = api.grpo_advantage(b.rewards, b.group_offsets, p, flags=flags)
    state = api.controller_init(p)
    w, coef, alpha = api.controller_step(state, p, disc, b.mask, b.seq_offsets, b.group_offsets, adv, flags=flags)
    grad, tl, loss = api.loss_grad_logits(logits, b.ids, b.mask, lse, None, coef, p.clip_eps, V=b.N, flags=flags)
    torch.cuda.synchronize()
    assert api.read_flags(flags) == 0
    # O(T) stages, stage-isolated on the GPU's log-probs
    mask, so, go = host(b.mask), host(b.seq_offsets), host(b.group_offsets)
    mu = host(b.logp_mu).astype(np.float64)
    lr, d, seq, grp, batch, _ = O.seq_discrepancy(host(logp).astype(np.float64), mu, mask, so, go,
                                                  host(ent).astype(np.float64))
    compare_seq(disc.seq_host(), seq)
    compare_batch(disc.batch_host(), batch)
    oadv = O.grpo_advantage(host(b.rewards).astype(np.float64), go, op)
    ow, oalpha, ost, info, _ = O.controller_step(O.controller_init(op), op, lr, mask, so, go, seq, grp, batch, oadv)
    assert_close_rel(host(w), ow, floor=1e-7, what="weight")
    ocoef = O.loss_coefficients(ow, oadv, mask, so, seq, grp, batch, op)
    tl_ref, loss_ref = O.surrogate_loss(host(logp).astype(np.float64), None, oadv, ow, mask, so, seq, grp, batch, op)
    assert_loss(float(loss), loss_ref, tl_ref)
    # vocabulary-wide outputs on sampled rows, from the oracle's own fp64 logits: 1,024 random rows and the first
    # and last row of every 128-row tile (so every edge of the 32-tile bands too), in blocks of 256 rows
    rng = np.random.default_rng(3)
    starts = np.arange(0, b.T, 128)
    rows = np.unique(np.concatenate([rng.choice(b.T, size=1024, replace=False), starts,
                                     np.minimum(starts + 127, b.T - 1)]))
    assert len(rows) >= 1024 + 2 * len(starts) - 64
    Wf = _f64(b.weight)
    Wabs = np.abs(Wf)
    ids_h = host(b.ids)
    lse_h, logp_h, ent_h = host(lse), host(logp), host(ent)
    for k in range(0, len(rows), 256):
        rr = rows[k:k + 256]
        Hr = _f64(b.hidden[torch.as_tensor(rr, device=DEV)])
        z = O.lmhead_logits(Hr, Wf)
        _check_logits(logits[torch.as_tensor(rr, device=DEV), :b.N], z, np.abs(Hr) @ Wabs.T, b.K,
                      "logits (sampled rows)")
        olse, ologp, oH, _ = O.token_stats(z, ids_h[rr], mask[rr])
        # a stored logit one bf16 ulp off the oracle's rounding (both valid) moves lse by p_j |dz_j| and log p by
        # that plus |dz_a|: the statistics may differ from the oracle's chain by that much beyond TOL_LOGP
        zg = rows_f64(logits, rr, b.N)
        dz = np.abs(zg - z)
        shift = (np.exp(z - olse[:, None]) * dz).sum(axis=1)
        a = ids_h[rr]
        assert_close_abs(lse_h[rr], olse, TOL_LOGP + shift, "lse")
        assert_close_abs(logp_h[rr], ologp, TOL_LOGP + shift + dz[np.arange(len(rr)), a], "logp")
        assert_close_rel(ent_h[rr], oH, floor=1e-5, what="entropy")
        # The gradient pass is judged on the logits it consumed: a logit one bf16 ulp
        # away (about 0.1 % of them, see _check_logits) moves its p by e^ulp, ~1-2 %.
        glse, _, _, _ = O.token_stats(zg, ids_h[rr], mask[rr])
        lse_full = np.zeros(b.T)
        lse_full[rr] = glse
        ograd, _, _ = O.loss_grad_logits(zg, ids_h, mask, lse_full, None, oadv, ow, so, seq, grp, batch, op, rows=rr)
        assert_grad_rows(grad_rows(grad, rr, b.N), ograd, ocoef[rr], a)


def test_lmhead_flags_nonfinite_and_bad_id_rows_like_token_stats():
    """A NaN in one hidden row makes that row's logits NaN: the merge gives NaN
    lse/logp/entropy there and raises NONFINITE; an id outside [0, N) gives
    logp = 0 and BAD_ID; every other row is unaffected.  Same outputs and flags
    as acrl_token_stats on the stored logits."""
    M, N, K = 130, 520, 64
    gen = torch.Generator(device=DEV).manual_seed(11)
    H = torch.randn((M, K), generator=gen, device=DEV).to(torch.bfloat16)
    H[5, 17] = float("nan")
    Wt = (0.02 * torch.randn((N, K), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, N, (M,), generator=gen, device=DEV, dtype=torch.int32)
    ids[7] = N
    flags = api.new_flags()
    logits, partials = api.lmhead_logits_stats(H, Wt, N=N, flags=flags)
    lse, logp, ent = api.lmhead_merge(partials, logits, ids, None, N=N, flags=flags)
    f = api.read_flags(flags)
    assert f == (acrl.FLAG_NONFINITE | acrl.FLAG_BAD_ID)
    assert torch.isnan(logits[5, :N].float()).all() and not torch.isnan(logits[:5, :N].float()).any()
    for t in (lse, logp, ent):
        assert torch.isnan(t[5]) and torch.isfinite(t[:5]).all() and torch.isfinite(t[6:]).all()
    assert float(logp[7]) == 0.0
    flags2 = api.new_flags()
    lse2, logp2, ent2 = api.token_stats(logits, ids, None, V=N, flags=flags2)
    assert api.read_flags(flags2) == f
    ok = torch.ones(M, dtype=torch.bool, device=DEV)
    ok[5] = False
    assert_close_abs(host(lse[ok]), host(lse2[ok]), 1e-5 + 1e-6 * np.abs(host(lse2[ok])), "lse")
    assert_close_abs(host(logp[ok]), host(logp2[ok]), 2e-5, "logp")
    assert_close_rel(host(ent[ok]), host(ent2[ok]), rel=1e-4, floor=1e-6, what="entropy")
    assert torch.isnan(lse2[5]) and float(logp2[7]) == 0.0


def _managed_alloc(nbytes):
    """Managed memory from the driver API (cuMemAllocManaged, attached
    globally), for the operand-placement check; returns (address, free)."""
    import ctypes
    cu = ctypes.CDLL("libcuda.so.1")
    torch.cuda.synchronize()              # the runtime has made the primary context current on this thread
    p = ctypes.c_uint64(0)
    assert cu.cuMemAllocManaged(ctypes.byref(p), ctypes.c_size_t(nbytes), ctypes.c_uint(1)) == 0 and p.value
    return p.value, lambda: cu.cuMemFree_v2(ctypes.c_uint64(p.value))


def test_lmhead_refuses_operands_outside_this_gpu():
    """hidden, weight and logits must be plain device memory of the current
    device, since the GEMM's TMA copies are encoded over them: managed memory
    and host memory (page-locked or pageable) are refused on the host with
    ACRL_ERR_INVALID_ARG before anything is launched, by both LM-head entry
    points, and the context stays usable."""
    M, N, K = 130, 264, 64
    gen = torch.Generator(device=DEV).manual_seed(21)
    H = torch.randn((M, K), generator=gen, device=DEV).to(torch.bfloat16)
    Wt = (0.02 * torch.randn((N, K), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, N, (M,), generator=gen, device=DEV, dtype=torch.int32)
    logits = torch.full((M, N), 7.0, dtype=torch.bfloat16, device=DEV)
    partials = torch.empty(api.lmhead_workspace_bytes(M, N) // 4, dtype=torch.float32, device=DEV)
    out = [torch.full((M,), 3.0, device=DEV) for _ in range(3)]
    flags = api.new_flags()
    L = _abi.lib()
    stream = torch.cuda.current_stream().cuda_stream
    size = max(M, N) * max(K, N) * 2
    pinned = torch.empty(size // 2, dtype=torch.bfloat16, pin_memory=True)
    pageable = torch.empty(size // 2, dtype=torch.bfloat16)
    managed, free_managed = _managed_alloc(size)
    try:
        for bad in (managed, pinned.data_ptr(), pageable.data_ptr()):
            assert bad % 16 == 0
            for slot in range(3):
                ptrs = [H.data_ptr(), Wt.data_ptr(), logits.data_ptr()]
                ptrs[slot] = bad
                st = L.acrl_lmhead_logits_stats(ptrs[0], M, K, K, ptrs[1], N, K, ptrs[2], N, partials.data_ptr(),
                                                flags.data_ptr(), stream)
                assert st == _abi.ERR_INVALID_ARG, (hex(bad), slot, st)
                st = L.acrl_lmhead_stats_noalloc(ptrs[0], M, K, K, ptrs[1], N, K, ptrs[2], N, ids.data_ptr(), None,
                                                 out[0].data_ptr(), out[1].data_ptr(), out[2].data_ptr(),
                                                 flags.data_ptr(), stream)
                assert st == _abi.ERR_INVALID_ARG, (hex(bad), slot, st)
        torch.cuda.synchronize()
        # nothing ran: outputs untouched, no flag raised
        assert api.read_flags(flags) == 0
        assert bool((logits.float() == 7.0).all()) and all(bool((t == 3.0).all()) for t in out)
    finally:
        free_managed()
    # the same call on device memory runs, and the context is fine
    lg, part = api.lmhead_logits_stats(H, Wt, N=N, flags=flags)
    lse, logp, ent = api.lmhead_merge(part, lg, ids, None, N=N, flags=flags)
    assert api.read_flags(flags) == 0
    lse2, _, _ = api.token_stats(lg, ids, None, V=N)
    assert_close_abs(host(lse), host(lse2), 1e-5, "lse after the refusals")
