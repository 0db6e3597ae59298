"""ACRL vocabulary-wide hot path on one GB300 (sm_103a).

The computation lives in libacrl.so (hand-written CUDA behind the C ABI of
include/acrl.h).  This package is its Python binding: `api` has one function
per entry point, `pipeline.AcrlStep` runs the whole on-policy pass,
`pipeline.importance_weights` makes the weights from log-probs alone,
`pipeline.HostPipeline` runs the pass on host-memory batches,
`autograd.acrl_loss` exposes it to torch.autograd, and `build` compiles the
library.  Importing the package does not load the
library; the first call does, and fails loudly if it has not been built.
"""

from ._abi import (AGG_SEQ_MEAN_TOKEN_MEAN, AGG_TOKEN_MEAN, FLAG_BAD_ID, FLAG_BAD_OFFSETS, FLAG_NONFINITE,  # noqa: F401
                   FLAG_TIMEOUT,
                   FLAG_X_NONPOS, MODE_ACRL, MODE_ACRL_CONTINUOUS, MODE_ACRL_FALLBACK, MODE_MIS, MODE_NONE,
                   MODE_TIS, SINGLETON_MEAN0_STD1, SINGLETON_ZERO, Y_BATCH, Y_GROUP, Y_SEQUENCE, AcrlError, Params)
from .api import (controller_init, controller_step, grpo_advantage, loss_grad_logits, read_flags,  # noqa: F401
                  read_state, reduce_loss, seq_discrepancy, token_stats)
from .pipeline import AcrlStep, HostPipeline, Weights, importance_weights  # noqa: F401
from .autograd import acrl_loss  # noqa: F401

LIBRARY_NAME = "libacrl.so"
