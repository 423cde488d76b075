"""The in-register butterfly (tac_fwht_debug) against the dense Hadamard matrix of
the oracle: every basis vector for d <= 16 (brute force) and random rows for all d."""
import math

import numpy as np
import pytest

import parity

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("d", [2, 4, 8, 16, 32, 64, 128])
@pytest.mark.parametrize("dt", ["bf16", "fp32"])
def test_butterfly_matches_dense_hadamard(tac_gpu, orc, d, dt):
    import torch
    tac = tac_gpu
    words = tac.make_signs(5, 2, 1, d)
    s = parity.signs_pm1(words, d)
    rng = np.random.default_rng(d)
    x = rng.standard_normal((300, d)) * np.exp(rng.normal(0, 1, d))
    if d <= 16:
        x = np.concatenate([np.eye(d), -3.0 * np.eye(d), x])
    xt = torch.tensor(x, dtype=torch.float32)
    xt = (xt.to(torch.bfloat16) if dt == "bf16" else xt).cuda().contiguous()
    x64 = parity.to_f64(xt)
    y = tac.fwht_debug(xt, words, d)
    torch.cuda.synchronize()
    ref = orc.transform(x64, s)
    # fp32 butterfly: |dy| <= (log2 d + 1) u ||x||_1 / sqrt(d) (stages + final scaling)
    bound = (math.log2(d) + 2) * 2.0**-24 * np.abs(x64).sum(axis=1) / math.sqrt(d)
    err = np.abs(y.cpu().numpy().astype(np.float64) - ref)
    assert np.all(err <= bound[:, None] + 1e-45)
    if d in (4, 16, 64):  # 1/sqrt(d) exact: basis vectors come out exact
        nb = min(d, 16) if d <= 16 else 0
        assert np.array_equal(y.cpu().numpy()[:nb].astype(np.float64), ref[:nb])
