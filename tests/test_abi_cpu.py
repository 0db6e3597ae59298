"""The C-ABI library builds for sm_103a, loads, exports every function that
include/acrl.h declares, agrees with the binding on struct layouts, and
rejects bad host-side arguments before touching a GPU.  CPU only: no call
here launches a kernel."""

import ctypes
import shutil

import pytest

from paper_2607_24062_gb300 import _abi, build

pytestmark = pytest.mark.skipif(shutil.which("nvcc") is None and not build.up_to_date(),
                                reason="needs nvcc to build the library")


@pytest.fixture(scope="module")
def L():
    build.build()
    return _abi.lib()


def test_exports_every_declared_function(L):
    declared = _abi.header_functions()
    assert len(declared) >= 11
    for name in declared:
        assert hasattr(L, name), name
    assert set(declared) == set(_abi.SIGNATURES)


def test_binding_has_a_function_per_entry_point():
    """The binding mirrors the header: acrl_x is api.x, for every declaration."""
    from paper_2607_24062_gb300 import api
    missing = [n for n in _abi.header_functions() if not callable(getattr(api, n[len("acrl_"):], None))]
    assert not missing, missing


def test_abi_version_and_layouts(L):
    assert L.acrl_abi_version() == 2
    assert L.acrl_struct_size(0) == ctypes.sizeof(_abi.Params) == 64
    assert L.acrl_struct_size(1) == 48 and L.acrl_struct_size(2) == 64
    assert L.acrl_struct_size(3) == 24 and L.acrl_struct_size(4) == 104
    assert L.acrl_struct_size(99) == -1
    assert L.acrl_status_string(0) == b"ok" and L.acrl_status_string(1) == b"invalid argument"


def test_host_side_rejections(L):
    p = _abi.Params()
    bad = _abi.Params(C=1.0)
    E = _abi.ERR_INVALID_ARG
    fake = 0x1000  # never dereferenced: every call below is rejected on the host
    # token stats: ld < V, ld not a multiple of 8, misaligned logits, null outputs
    assert L.acrl_token_stats(fake, 4, 16, 8, fake, None, fake, fake, fake, fake, None) == E
    assert L.acrl_token_stats(fake, 4, 16, 20, fake, None, fake, fake, fake, fake, None) == E
    assert L.acrl_token_stats(fake + 2, 4, 16, 16, fake, None, fake, fake, fake, fake, None) == E
    assert L.acrl_token_stats(fake, 4, 16, 16, fake, None, None, fake, fake, fake, None) == E
    assert L.acrl_token_stats(fake, -1, 16, 16, fake, None, fake, fake, fake, fake, None) == E
    # V above 2^30 (column indices must stay in 32-bit range), for every vocabulary-wide call
    big = (1 << 30) + 8
    assert L.acrl_token_stats(fake, 4, big, big, fake, None, fake, fake, fake, fake, None) == E
    assert L.acrl_loss_grad_logits(fake, 4, big, big, fake, None, fake, None, fake, None, None, 0.2, fake, fake, fake,
                                   fake, None) == E
    # T = 0 is a valid no-op
    assert L.acrl_token_stats(None, 0, 16, 16, None, None, None, None, None, None, None) == _abi.OK
    # hyper-parameters out of range
    assert L.acrl_grpo_advantage(fake, fake, 1, 1, ctypes.byref(bad), fake, fake, None) == E
    assert L.acrl_controller_init(None, ctypes.byref(p), None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(gamma=0.0)), None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(calib_steps=0)), None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(mode=7)), None) == E
    # loss/grad: clip eps out of range, misaligned grad
    assert L.acrl_loss_grad_logits(fake, 4, 16, 16, fake, None, None, None, fake, None, None, 1.5, fake, fake, fake,
                                   fake, None) == E
    assert L.acrl_loss_grad_logits(fake, 4, 16, 16, fake, None, None, None, fake, None, None, 0.2, fake + 8, fake,
                                   fake, fake, None) == E
    # the entropy bonus needs both the entropies and their coefficients
    assert L.acrl_loss_grad_logits(fake, 4, 16, 16, fake, None, None, None, fake, fake, None, 0.2, fake, fake, fake,
                                   fake, None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(kappa=0.0)), None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(x_ema=1.5)), None) == E
    assert L.acrl_controller_init(fake, ctypes.byref(_abi.Params(entropy_coeff=-1.0)), None) == E
    assert L.acrl_read_flags(None, None, None) == E
    # the host-buffer pipeline: shapes, workspace and handle checked before any CUDA call
    assert L.acrl_host_pipeline_workspace_bytes(0, 16, 1, 1, 1) == -1
    assert L.acrl_host_pipeline_workspace_bytes(4, 16, 1, 1, 5000) == -1
    ws = L.acrl_host_pipeline_workspace_bytes(64, 16, 2, 1, 4)
    assert ws > 64 * 16 * 2
    h = ctypes.c_void_p()
    assert L.acrl_host_pipeline_create(None, 64, 16, 16, 2, 1, 4, fake, ws) == E
    assert L.acrl_host_pipeline_create(ctypes.byref(h), 64, 16, 12, 2, 1, 4, fake, ws) == E       # ld < V
    assert L.acrl_host_pipeline_create(ctypes.byref(h), 3, 16, 16, 2, 1, 4, fake, ws) == E        # chunks > T
    assert L.acrl_host_pipeline_create(ctypes.byref(h), 64, 16, 16, 2, 1, 4, fake, ws - 1) == E   # too small
    assert L.acrl_host_pipeline_create(ctypes.byref(h), 64, 16, 16, 2, 1, 4, fake + 8, ws) == E   # misaligned
    assert h.value is None
    assert L.acrl_host_pipeline_step(None, ctypes.byref(p), fake, fake, fake, None, fake, fake, fake, fake, fake,
                                     fake, fake, None) == E
    assert L.acrl_host_pipeline_destroy(None) == E
    assert L.acrl_host_pipeline_begin(None, fake, fake, None, fake, fake, fake, fake, fake, None) == E
    assert L.acrl_host_pipeline_finish(None, ctypes.byref(p), fake, fake, fake, fake, None) == E
    assert L.acrl_host_pipeline_batch_stats(None) is None
    assert L.acrl_controller_save(None, fake, None) == E and L.acrl_controller_save(fake, None, None) == E
    assert L.acrl_controller_load(None, fake, None) == E and L.acrl_controller_load(fake, None, None) == E
    assert L.acrl_reduce_loss(None, 4, fake, None) == E
    assert L.acrl_selftest_wait_timeout(None, 1000, None) == E
    assert L.acrl_selftest_wait_timeout(fake, 3_000_000_000, None) == E
    # the LM-head calls encode their tensor-core copies over hidden, weight and logits, which must be device memory
    # of the current device: pointers that cannot be shown to be (here: no device, or a host address) are refused
    # before anything is launched
    assert L.acrl_lmhead_logits_stats(fake, 4, 64, 64, fake, 256, 64, fake, 256, fake, fake, None) == E
    assert L.acrl_lmhead_stats_noalloc(fake, 4, 64, 64, fake, 256, 64, fake, 256, fake, None, fake, fake, fake, fake,
                                       None) == E


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(_abi, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(_abi, "_LIB", None)
    with pytest.raises(_abi.AcrlError):
        _abi.lib()


def test_binding_rejects_buffers_on_different_devices():
    """Every buffer of one call must be on one GPU: the binding refuses a mix
    before any pointer reaches the library (checked here with host and meta
    tensors, so no GPU is needed)."""
    import torch
    from paper_2607_24062_gb300 import api
    a, b = torch.empty(4), torch.empty(4, device="meta")
    with pytest.raises(api.AcrlError, match="one GPU"):
        api._one_device((a, None, b))
    with pytest.raises(api.AcrlError, match="CUDA"):
        api._one_device((a, a))
    with pytest.raises(api.AcrlError, match="CUDA"):
        api._one_device((None,))


def test_kernels_do_not_spill_and_fit_their_occupancy(L):
    """The build's ptxas report: no kernel spills registers to local memory,
    and the gradient kernels stay within the register counts their CTAs per
    SM rely on (two 768-thread streaming CTAs need at most 42 registers a
    thread, two 512-thread recompute CTAs at most 64)."""
    import os
    import re
    path = os.path.join(build.BUILD, "ptxas.txt")
    if not os.path.exists(path):
        build.build(force=True)
    text = open(path).read()
    spills = re.findall(r"(\d+) bytes spill stores, (\d+) bytes spill loads", text)
    assert spills, "no ptxas resource report"
    assert all(int(a) == 0 and int(b) == 0 for a, b in spills), spills
    regs = {}
    name = None
    for line in text.splitlines():
        m = re.search(r"Compiling entry function '(\S+)'", line)
        if m:
            name = m.group(1)
            continue
        m = re.search(r"Used (\d+) registers", line)
        if m and name:
            regs[name] = int(m.group(1))
            name = None
    limits = {r"loss_grad_ctaILi768ELi4ELb0E": 42, r"loss_grad_ctaILi512ELi4ELb1E": 64}
    for pattern, limit in limits.items():
        found = {k: v for k, v in regs.items() if re.search(pattern, k)}
        assert found, pattern
        assert all(v <= limit for v in found.values()), found
