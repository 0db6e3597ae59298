"""acrl_lmhead_stats_noalloc against the workspace path.

Some callers of this library cannot allocate device memory: a plugin that a
framework hands only tensors while its caching allocator owns nearly all of
HBM, or a step that must not call cudaMalloc/cudaFree.  For them the LM-head
GEMM + merge has an entry point whose scratch is a fixed 16 MiB device array
inside the library.  This test calls it through the C ABI twice in a row, on
two different problems, and checks each result bit for bit against
acrl_lmhead_logits_stats + acrl_lmhead_merge with a caller-provided
workspace (the same kernels in the same fixed reduction order); it also
checks that an oversized problem is refused on the host.  It lives in a file
of its own, collected last, and passes alone or after the rest of the
suite."""

import pytest
import torch

pytestmark = pytest.mark.gpu

from paper_2607_24062_gb300 import _abi, api  # noqa: E402

DEV = "cuda"


def _noalloc(H, Wt, N, ids, mask):
    M, K = H.shape
    ldl = ((N + 7) // 8) * 8
    logits = torch.empty((M, ldl), dtype=torch.bfloat16, device=DEV)
    lse, logp, ent = (torch.empty(M, dtype=torch.float32, device=DEV) for _ in range(3))
    flags = api.new_flags()
    st = _abi.lib().acrl_lmhead_stats_noalloc(H.data_ptr(), M, K, H.stride(0), Wt.data_ptr(), N, Wt.stride(0),
                                              logits.data_ptr(), ldl, ids.data_ptr(),
                                              None if mask is None else mask.data_ptr(), lse.data_ptr(),
                                              logp.data_ptr(), ent.data_ptr(), flags.data_ptr(),
                                              torch.cuda.current_stream().cuda_stream)
    _abi.check(st, "acrl_lmhead_stats_noalloc")
    return logits, lse, logp, ent, flags


def _problem(M, N, K, seed):
    gen = torch.Generator(device=DEV).manual_seed(seed)
    H = torch.randn((M, K), generator=gen, device=DEV).to(torch.bfloat16)
    Wt = (0.02 * torch.randn((N, K), generator=gen, device=DEV)).to(torch.bfloat16)
    ids = torch.randint(0, N, (M,), generator=gen, device=DEV, dtype=torch.int32)
    mask = (torch.rand(M, generator=gen, device=DEV) < 0.95).to(torch.uint8)
    return H, Wt, ids, mask


def test_noalloc_matches_workspace_path_twice():
    for (M, N, K, seed) in [(1000, 32000, 512, 1), (1765, 151936, 1024, 2)]:
        H, Wt, ids, mask = _problem(M, N, K, seed)
        logits, lse, logp, ent, flags = _noalloc(H, Wt, N, ids, mask)
        ref_logits, part = api.lmhead_logits_stats(H, Wt, N=N)
        rlse, rlogp, rent = api.lmhead_merge(part, ref_logits, ids, mask, N=N)
        torch.cuda.synchronize()
        assert api.read_flags(flags) == 0
        # the same kernels with the same fixed reduction order: every output bit for bit (a partial state
        # that another call's use of the shared array had shifted would show here)
        assert torch.equal(logits[:, :N].view(torch.int16), ref_logits[:, :N].view(torch.int16))
        for got, ref, what in ((lse, rlse, "lse"), (logp, rlogp, "logp"), (ent, rent, "entropy")):
            assert torch.equal(got.view(torch.int32), ref.view(torch.int32)), what


def test_noalloc_refuses_oversized_problem():
    H, Wt, ids, mask = _problem(1766, 151936, 64, 3)   # one row more than 16 MiB of partial states holds
    st = _abi.lib().acrl_lmhead_stats_noalloc(H.data_ptr(), 1766, 64, 64, Wt.data_ptr(), 151936, 64,
                                              H.data_ptr(), 151936, ids.data_ptr(), None, H.data_ptr(),
                                              H.data_ptr(), H.data_ptr(), api.new_flags().data_ptr(), None)
    assert st == _abi.ERR_SCRATCH_TOO_SMALL
    assert b"scratch" in _abi.lib().acrl_status_string(st)


def test_noalloc_through_the_binding():
    H, Wt, ids, mask = _problem(300, 2000, 72, 5)
    logits, lse, logp, ent = api.lmhead_stats_noalloc(H, Wt, ids, mask, N=2000)
    logits2, lse2, logp2, ent2, _ = _noalloc(H, Wt, 2000, ids, mask)
    torch.cuda.synchronize()
    assert torch.equal(logits[:, :2000], logits2[:, :2000])
    for a, b in ((lse, lse2), (logp, logp2), (ent, ent2)):
        assert torch.equal(a, b)
