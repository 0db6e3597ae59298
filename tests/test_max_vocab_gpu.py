"""The largest vocabulary the library accepts (V = 2^30 columns, one 2 GB
bf16 row each), checked through closed forms that hold at any size rather
than through the oracle (a float64 copy of such rows would need 8 GB each):

- a constant row is uniform: lse = ln V, log p = -ln V, H = ln V;
- a row of zeros with one entry c: S = V - 1 + e^c, lse = ln S,
  log p(c) = c - ln S, H = ln S - c e^c / S;
- dL/dlogits = coef (p - onehot) sums to 0 over each row, the on-policy token
  loss is -coef (r = 1), and masked or zero-coefficient rows are 0.
"""

import math

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

import paper_2607_24062_gb300 as acrl  # noqa: E402
from paper_2607_24062_gb300 import api  # noqa: E402

V = 1 << 30
J0, C = 123_456_789, 10.0


def test_max_vocabulary_closed_forms():
    dev = torch.device("cuda")
    T = 4
    logits = torch.zeros((T, V), dtype=torch.bfloat16, device=dev)
    logits[1, J0] = C
    ids = torch.tensor([V - 1, J0, 7, 5], dtype=torch.int32, device=dev)
    mask = torch.tensor([1, 1, 0, 1], dtype=torch.uint8, device=dev)
    flags = api.new_flags(dev)
    lse, logp, H = api.token_stats(logits, ids, mask, V=V, flags=flags)
    lse_h, logp_h, H_h = lse.cpu().numpy(), logp.cpu().numpy(), H.cpu().numpy()

    lnV = 30 * math.log(2.0)
    S = (V - 1) + math.exp(C)
    for t, (l, lp, h) in {0: (lnV, -lnV, lnV), 3: (lnV, -lnV, lnV),
                          1: (math.log(S), C - math.log(S), math.log(S) - C * math.exp(C) / S)}.items():
        assert abs(lse_h[t] - l) <= 2e-4 and abs(logp_h[t] - lp) <= 2e-4, t
        assert abs(H_h[t] - h) <= 1e-3 * h, t
    assert lse_h[2] == 0.0 and logp_h[2] == 0.0 and H_h[2] == 0.0

    coef = torch.tensor([0.5, -2.0, 1.0, 0.0], dtype=torch.float32, device=dev)
    grad, token_loss, loss = api.loss_grad_logits(logits, ids, mask, lse, None, coef, 0.2, V=V, flags=flags)
    assert api.read_flags(flags) == 0

    cols = torch.tensor([0, 1, J0 - 1, J0, J0 + 1, V // 2, V - 2, V - 1], dtype=torch.int64, device=dev)
    g = grad[:, cols].float().cpu().numpy()
    p0 = 1.0 / V
    want0 = 0.5 * np.array([p0] * 7 + [p0 - 1.0])
    np.testing.assert_allclose(g[0], want0, rtol=1e-2)
    pz, pc = 1.0 / S, math.exp(C) / S
    want1 = -2.0 * np.array([pz, pz, pz, pc - 1.0, pz, pz, pz, pz])
    np.testing.assert_allclose(g[1], want1, rtol=1e-2)
    assert not g[2].any() and not g[3].any()
    # every row sums to 0; the masked and zero-coefficient rows are 0 everywhere
    for t in range(T):
        row = grad[t, :V]
        assert abs(float(torch.sum(row, dtype=torch.float64))) <= 1e-2 * abs(float(coef[t])) + 1e-30, t
    assert int(torch.count_nonzero(grad[2])) == 0 and int(torch.count_nonzero(grad[3])) == 0

    tl = token_loss.cpu().numpy()
    np.testing.assert_allclose(tl, [-0.5, 2.0, 0.0, 0.0], rtol=1e-6)
    assert float(loss) == pytest.approx(float(tl.sum()), rel=1e-6)
