"""The host-buffer pipeline (acrl_host_pipeline_*) against the device calls:
batches held in page-locked host memory, uploaded and processed in uneven
row chunks with the gradient downloaded chunk by chunk, must give the
gradient, the loss, the flags and the controller state of AcrlStep on the
same data bit for bit, over consecutive steps (the first one calibrates X)
that overlap on the copy streams."""

import numpy as np
import pytest
import torch

import workloads as W

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import api  # noqa: E402

DEV = "cuda"


def _pinned(t):
    h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
    h.copy_(t)
    return h


@pytest.mark.parametrize("case", ["padded", "no_mask", "entropy_bonus", "one_chunk"])
def test_host_pipeline_matches_device_calls(case):
    if case == "no_mask":
        spec = W.small_variant(W.TINY, name="hp_nomask", n_prompts=3, group_size=2, len_lo=40, len_hi=90, V=20011)
    else:
        spec = W.small_variant(W.GRPO, name="hp", n_prompts=3, group_size=4, len_lo=20, len_hi=120, V=20011,
                               pad_multiple=16, ld_pad=8)
    b = W.generate(spec, seed=41, device=DEV)
    mask = None if case == "no_mask" else b.mask
    if case == "no_mask":
        assert bool(b.mask.all())
    p = acrl.Params(entropy_coeff=0.01 if case == "entropy_bonus" else 0.0)
    chunks = 1 if case == "one_chunk" else 7          # uneven chunks, more than the four-slot gradient ring

    ref = acrl.AcrlStep.for_batch(b, p)
    hp = acrl.HostPipeline(b.T, b.V, b.ld, b.S, b.Gn, chunks=chunks)
    state = api.controller_init(p)
    flags = api.new_flags()
    h = {k: _pinned(getattr(b, k)) for k in ("logits", "ids", "logp_mu", "rewards", "seq_offsets", "group_offsets")}
    h_mask = None if mask is None else _pinned(mask)
    grads = [torch.zeros((b.T, b.ld), dtype=torch.bfloat16, pin_memory=True) for _ in range(3)]
    losses = [torch.zeros(1, dtype=torch.float32, pin_memory=True) for _ in range(3)]
    for k in range(3):                                # enqueued back to back: the steps overlap
        hp.step(state, p, h["logits"], h["ids"], h_mask, h["logp_mu"], h["rewards"], h["seq_offsets"],
                h["group_offsets"], grads[k], losses[k], flags)
    torch.cuda.synchronize()
    for k in range(3):
        ref.run(b.logits, b.ids, mask, b.logp_mu, b.rewards, b.seq_offsets, b.group_offsets)
        torch.cuda.synchronize()
        g_ref = ref.grad[:, : b.V].cpu()
        assert torch.equal(grads[k][:, : b.V].view(torch.int16), g_ref.view(torch.int16)), f"grad, step {k}"
        assert float(losses[k][0]) == float(ref.loss[0]), f"loss, step {k}"
    assert api.read_flags(flags) == api.read_flags(ref.flags)
    assert api.save_state(state) == api.save_state(ref.state)
    hp.close()


def test_host_pipeline_rejects_device_tensors_and_wrong_shapes():
    spec = W.small_variant(W.TINY, name="hp_bad", n_prompts=2, group_size=2, len_lo=16, len_hi=16, V=4096)
    b = W.generate(spec, seed=3, device=DEV)
    p = acrl.Params()
    hp = acrl.HostPipeline(b.T, b.V, b.ld, b.S, b.Gn, chunks=2)
    state, flags = api.controller_init(p), api.new_flags()
    grad = torch.zeros((b.T, b.ld), dtype=torch.bfloat16)
    loss = torch.zeros(1)
    with pytest.raises(acrl.AcrlError):   # device logits where host memory is required
        hp.step(state, p, b.logits, b.ids.cpu(), None, b.logp_mu.cpu(), b.rewards.cpu(), b.seq_offsets.cpu(),
                b.group_offsets.cpu(), grad, loss, flags)
    with pytest.raises(acrl.AcrlError):   # a gradient buffer of the wrong shape
        hp.step(state, p, b.logits.cpu(), b.ids.cpu(), None, b.logp_mu.cpu(), b.rewards.cpu(), b.seq_offsets.cpu(),
                b.group_offsets.cpu(), grad[:-1], loss, flags)
    hp.close()
    with pytest.raises(acrl.AcrlError):   # closed
        hp.step(state, p, b.logits.cpu(), b.ids.cpu(), None, b.logp_mu.cpu(), b.rewards.cpu(), b.seq_offsets.cpu(),
                b.group_offsets.cpu(), grad, loss, flags)
    assert np.isfinite(float(loss[0]))


def test_host_pipeline_exchange_matches_device_calls():
    """The two-phase step (begin, the batch-statistics exchange, finish) with an
    exchange that doubles the three summed fields, as an all-reduce over two
    ranks holding the same batch would: the same results as AcrlStep with the
    same exchange, bit for bit, over two steps."""
    from paper_2607_24062_gb300 import distributed as D

    def as_two_ranks(buf):
        for name, dt in (("n_tokens", torch.int64), ("n_groups_valid", torch.int32), ("Y_sum", torch.float64)):
            D._field(buf, name, dt).mul_(2)

    spec = W.small_variant(W.GRPO, name="hp_x", n_prompts=3, group_size=4, len_lo=20, len_hi=120, V=3000,
                           perturb_frac=0.4, perturb_std=0.3)
    b = W.generate(spec, seed=43, device=DEV)
    p = acrl.Params()
    ref = acrl.AcrlStep.for_batch(b, p)
    hp = acrl.HostPipeline(b.T, b.V, b.ld, b.S, b.Gn, chunks=5)
    state, flags = api.controller_init(p), api.new_flags()
    h = {k: _pinned(getattr(b, k)) for k in ("logits", "ids", "mask", "logp_mu", "rewards", "seq_offsets",
                                             "group_offsets")}
    for k in range(2):
        grad = torch.zeros((b.T, b.ld), dtype=torch.bfloat16, pin_memory=True)
        loss = torch.zeros(1, dtype=torch.float32, pin_memory=True)
        hp.step(state, p, h["logits"], h["ids"], h["mask"], h["logp_mu"], h["rewards"], h["seq_offsets"],
                h["group_offsets"], grad, loss, flags, exchange=as_two_ranks)
        ref.run_batch(b, exchange=as_two_ranks)
        torch.cuda.synchronize()
        assert torch.equal(grad[:, : b.V].view(torch.int16), ref.grad[:, : b.V].cpu().view(torch.int16)), k
        assert float(loss[0]) == float(ref.loss[0])
        bs = api.read_structs(hp.batch_stats(), acrl.api.BATCH_DTYPE, 1)[0]
        assert int(bs["n_groups_valid"]) == 2 * b.Gn
    assert api.save_state(state) == api.save_state(ref.state)
    hp.close()


def test_host_pipeline_different_batches_back_to_back():
    """Four steps on four different batches of one shape, enqueued back to
    back from four sets of host buffers: every upload of step k+1 lands while
    step k still computes and downloads, so a missing order between them would
    mix batches.  Each step must equal AcrlStep run on that step's batch."""
    spec = W.small_variant(W.GRPO, name="hp_seq", n_prompts=3, group_size=4, len_lo=20, len_hi=150, V=8000,
                           pad_multiple=16)
    b = W.generate(spec, seed=47, device=DEV)
    p = acrl.Params()
    n = 4
    gen = torch.Generator(device=DEV).manual_seed(5)
    logits = [(3.0 * torch.randn((b.T, b.ld), generator=gen, device=DEV)).to(torch.bfloat16) for _ in range(n)]
    mus = [(b.logp_mu + 0.05 * torch.randn(b.T, generator=gen, device=DEV)).clamp(max=0.0) for _ in range(n)]
    rewards = [(torch.rand(b.S, generator=gen, device=DEV) < 0.4).float() for _ in range(n)]
    hp = acrl.HostPipeline(b.T, b.V, b.ld, b.S, b.Gn, chunks=6)
    state, flags = api.controller_init(p), api.new_flags()
    small = {k: _pinned(getattr(b, k)) for k in ("ids", "mask", "seq_offsets", "group_offsets")}
    h_logits = [_pinned(z) for z in logits]
    h_mu = [_pinned(m) for m in mus]
    h_r = [_pinned(r) for r in rewards]
    grads = [torch.zeros((b.T, b.ld), dtype=torch.bfloat16, pin_memory=True) for _ in range(n)]
    losses = [torch.zeros(1, dtype=torch.float32, pin_memory=True) for _ in range(n)]
    for k in range(n):
        hp.step(state, p, h_logits[k], small["ids"], small["mask"], h_mu[k], h_r[k], small["seq_offsets"],
                small["group_offsets"], grads[k], losses[k], flags)
    torch.cuda.synchronize()
    ref = acrl.AcrlStep.for_batch(b, p)
    for k in range(n):
        ref.run(logits[k], b.ids, b.mask, mus[k], rewards[k], b.seq_offsets, b.group_offsets)
        torch.cuda.synchronize()
        assert torch.equal(grads[k][:, : b.V].view(torch.int16), ref.grad[:, : b.V].cpu().view(torch.int16)), k
        assert float(losses[k][0]) == float(ref.loss[0]), k
    assert api.save_state(state) == api.save_state(ref.state)
    hp.close()
