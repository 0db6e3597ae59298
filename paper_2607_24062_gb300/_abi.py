"""ctypes declarations of the C ABI in include/acrl.h and the struct layouts.

Loading fails loudly when the library has not been built: there is no
fallback implementation anywhere in this package.
"""

from __future__ import annotations

import ctypes
import os
import re

import numpy as np

PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG, "libacrl.so")
HEADER = os.path.join(os.path.dirname(PKG), "include", "acrl.h")

c_i32, c_i64, c_f32, c_f64, c_p = ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_double, ctypes.c_void_p

# status codes, flag bits and enums (values fixed by include/acrl.h)
OK, ERR_INVALID_ARG, ERR_CUDA, ERR_NOT_IMPLEMENTED, ERR_DEVICE_FLAGS, ERR_SCRATCH_TOO_SMALL = 0, 1, 2, 3, 4, 5
FLAG_BAD_ID, FLAG_NONFINITE, FLAG_BAD_OFFSETS, FLAG_X_NONPOS, FLAG_TIMEOUT = 0x1, 0x2, 0x4, 0x8, 0x10
MODE_NONE, MODE_TIS, MODE_MIS, MODE_ACRL, MODE_ACRL_CONTINUOUS, MODE_ACRL_FALLBACK = 0, 1, 2, 3, 4, 5
Y_GROUP, Y_SEQUENCE, Y_BATCH = 0, 1, 2
AGG_SEQ_MEAN_TOKEN_MEAN, AGG_TOKEN_MEAN = 0, 1
SINGLETON_MEAN0_STD1, SINGLETON_ZERO = 0, 1


class Params(ctypes.Structure):
    """acrl_params.  Defaults: gamma 0.65 and C 3 as in Sec. 5.1 of the paper."""

    _fields_ = [("gamma", c_f32), ("C", c_f32), ("clip_eps", c_f32), ("adv_eps", c_f32), ("kappa", c_f32),
                ("x_ema", c_f32), ("entropy_coeff", c_f32), ("reserved", c_f32), ("mode", c_i32),
                ("y_gran", c_i32), ("agg", c_i32), ("adv_ddof", c_i32), ("singleton_rule", c_i32),
                ("calib_steps", c_i32), ("X_init", c_f64)]

    def __init__(self, gamma=0.65, C=3.0, clip_eps=0.2, adv_eps=1e-6, kappa=1.0, x_ema=0.0, entropy_coeff=0.0,
                 mode=MODE_ACRL, y_gran=Y_GROUP, agg=AGG_SEQ_MEAN_TOKEN_MEAN, adv_ddof=1,
                 singleton_rule=SINGLETON_MEAN0_STD1, calib_steps=1, X_init=0.0):
        super().__init__(gamma, C, clip_eps, adv_eps, kappa, x_ema, entropy_coeff, 0.0, mode, y_gran, agg, adv_ddof,
                         singleton_rule, calib_steps, X_init)

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


STATE_DTYPE = np.dtype([("X", "<f8"), ("calib_sum", "<f8"), ("calib_count", "<i8"), ("step", "<i8"),
                        ("calib_done", "<i4"), ("calibrated", "<i4"), ("flags", "<i4"), ("reserved", "<i4")])
SEQ_DTYPE = np.dtype([("n", "<i4"), ("group", "<i4"), ("mean_d", "<f4"), ("max_d", "<f4"), ("sum_d", "<f8"),
                      ("sum_d2", "<f8"), ("sum_lr", "<f8"), ("sum_H", "<f8"), ("sum_w", "<f8"),
                      ("n_trunc", "<i4"), ("alpha", "<f4")])
GRP_DTYPE = np.dtype([("n_valid_seqs", "<i4"), ("n_seqs", "<i4"), ("n_tokens", "<i8"), ("Y", "<f8")])
BATCH_DTYPE = np.dtype([("n_tokens", "<i8"), ("n_seqs_valid", "<i4"), ("n_groups_valid", "<i4"),
                        ("d_mean", "<f8"), ("d_max", "<f8"), ("d_std", "<f8"), ("Y_sum", "<f8"), ("Y_mean", "<f8"),
                        ("H_mean", "<f8"), ("lr_mean", "<f8"), ("X", "<f8"), ("trunc_frac", "<f8"),
                        ("w_mean", "<f8"), ("alpha_mean", "<f8")])

# name -> (restype, argtypes) for every entry point
SIGNATURES = {
    "acrl_status_string": (ctypes.c_char_p, [c_i32]),
    "acrl_abi_version": (c_i32, []),
    "acrl_struct_size": (c_i64, [c_i32]),
    "acrl_token_stats": (c_i32, [c_p, c_i64, c_i64, c_i64, c_p, c_p, c_p, c_p, c_p, c_p, c_p]),
    "acrl_seq_discrepancy": (c_i32, [c_p, c_p, c_p, c_i64, c_p, c_i32, c_p, c_i32, c_p, c_p, c_p, c_p, c_p, c_p,
                                     c_p, c_p]),
    "acrl_grpo_advantage": (c_i32, [c_p, c_p, c_i32, c_i32, ctypes.POINTER(Params), c_p, c_p, c_p]),
    "acrl_controller_init": (c_i32, [c_p, ctypes.POINTER(Params), c_p]),
    "acrl_controller_save": (c_i32, [c_p, c_p, c_p]),
    "acrl_controller_load": (c_i32, [c_p, c_p, c_p]),
    "acrl_controller_step": (c_i32, [c_p, ctypes.POINTER(Params), c_p, c_p, c_i64, c_p, c_i32, c_p, c_i32, c_p, c_p,
                                     c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p]),
    "acrl_loss_grad_logits": (c_i32, [c_p, c_i64, c_i64, c_i64, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_f32, c_p, c_p,
                                      c_p, c_p, c_p]),
    "acrl_reduce_loss": (c_i32, [c_p, c_i64, c_p, c_p]),
    "acrl_host_pipeline_workspace_bytes": (c_i64, [c_i64, c_i64, c_i32, c_i32, c_i32]),
    "acrl_host_pipeline_create": (c_i32, [ctypes.POINTER(c_p), c_i64, c_i64, c_i64, c_i32, c_i32, c_i32, c_p,
                                          c_i64]),
    "acrl_host_pipeline_step": (c_i32, [c_p, ctypes.POINTER(Params), c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p,
                                        c_p, c_p, c_p]),
    "acrl_host_pipeline_begin": (c_i32, [c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p, c_p]),
    "acrl_host_pipeline_finish": (c_i32, [c_p, ctypes.POINTER(Params), c_p, c_p, c_p, c_p, c_p]),
    "acrl_host_pipeline_batch_stats": (c_p, [c_p]),
    "acrl_host_pipeline_destroy": (c_i32, [c_p]),
    "acrl_lmhead_workspace_bytes": (c_i64, [c_i64, c_i64]),
    "acrl_lmhead_logits_stats": (c_i32, [c_p, c_i64, c_i64, c_i64, c_p, c_i64, c_i64, c_p, c_i64, c_p, c_p, c_p]),
    "acrl_lmhead_merge": (c_i32, [c_p, c_p, c_i64, c_i64, c_i64, c_p, c_p, c_p, c_p, c_p, c_p, c_p]),
    "acrl_lmhead_stats_noalloc": (c_i32, [c_p, c_i64, c_i64, c_i64, c_p, c_i64, c_i64, c_p, c_i64, c_p, c_p, c_p,
                                          c_p, c_p, c_p, c_p]),
    "acrl_read_flags": (c_i32, [c_p, ctypes.POINTER(c_i32), c_p]),
    "acrl_check_flags": (c_i32, [c_p, c_p]),
    "acrl_selftest_wait_timeout": (c_i32, [c_p, c_i64, c_p]),
}


def header_functions() -> list[str]:
    """Names of the functions declared in include/acrl.h."""
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\**\s+\**(acrl_[a-z_0-9]+)\s*\(",
                                 text, flags=re.M)))


class AcrlError(RuntimeError):
    pass


_LIB = None


def lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise AcrlError(f"{LIB_PATH} is missing: build it with "
                            "`python -c 'import __graft_entry__ as g; g.build()'` (needs nvcc)")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        sizes = {0: ctypes.sizeof(Params), 1: STATE_DTYPE.itemsize, 2: SEQ_DTYPE.itemsize, 3: GRP_DTYPE.itemsize,
                 4: BATCH_DTYPE.itemsize}
        for k, v in sizes.items():
            got = L.acrl_struct_size(k)
            if got != v:
                raise AcrlError(f"struct {k}: library size {got} != binding size {v}")
        _LIB = L
    return _LIB


def check(status: int, what: str):
    if status != OK:
        msg = lib().acrl_status_string(status).decode()
        raise AcrlError(f"{what}: {msg} (status {status})")
