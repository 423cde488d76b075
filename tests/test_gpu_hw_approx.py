"""The hardware approximations the encoder's certification relies on, measured
exhaustively over whole binades against correctly rounded references.

The encoder decides each angle code by a rigorous bound and each norm code by a
band that adds a full bound on its own arithmetic; those bounds assume a
relative error of at most parity.E_SQRT (2^-23, one ulp) for the hardware
square root, 2^-23 for the reciprocal, and for the base-2 logarithm an absolute
error of at most 2^-22 on [1/2, 2) and of 2^-22 plus 4u times the result
elsewhere (u = 2^-24).  The square root and the
reciprocal act on the exponent separately from the significand, so every input
of [1, 4) (sqrt) and [1, 2) (rcp) covers all normal inputs; lg2 is checked over
[1/2, 2) and on every binade at 4096 points each."""
import numpy as np
import pytest

import parity

pytestmark = pytest.mark.gpu


def _all_floats(lo: float, hi: float) -> np.ndarray:
    a = np.array([lo, hi], dtype=np.float32).view(np.uint32)
    return np.arange(a[0], a[1], dtype=np.uint32).view(np.float32)


def _run(tac, op, x):
    import torch
    y = tac.hw_approx_debug(op, torch.from_numpy(x).cuda())
    torch.cuda.synchronize()
    return y.cpu().numpy().astype(np.float64)


def test_sqrt_relative_error_bound(tac_gpu):
    x = _all_floats(1.0, 4.0)
    want = np.sqrt(x.astype(np.float64))
    for op in (tac_gpu.HW_SQRT, tac_gpu.HW_SQRT_FTZ):
        rel = np.abs(_run(tac_gpu, op, x) - want) / want
        assert rel.max() <= parity.E_SQRT, (op, rel.max() / parity.U)
    # a sample over other binades (subnormal inputs excluded for the ftz form)
    xs = (_all_floats(1.0, 4.0)[::997].astype(np.float64)[None, :] * 4.0 ** np.arange(-60, 61)[:, None])
    xs = xs.astype(np.float32).reshape(-1)
    xs = xs[(xs > 2.0**-125) & np.isfinite(xs)]
    want = np.sqrt(xs.astype(np.float64))
    for op in (tac_gpu.HW_SQRT, tac_gpu.HW_SQRT_FTZ):
        rel = np.abs(_run(tac_gpu, op, xs) - want) / want
        assert rel.max() <= parity.E_SQRT, (op, rel.max() / parity.U)


def test_rcp_relative_error_bound(tac_gpu):
    x = _all_floats(1.0, 2.0)
    want = 1.0 / x.astype(np.float64)
    rel = np.abs(_run(tac_gpu, tac_gpu.HW_RCP_FTZ, x) - want) / want
    assert rel.max() <= 2.0**-23, rel.max() / parity.U


def test_lg2_absolute_error_bound(tac_gpu):
    x = _all_floats(0.5, 2.0)
    want = np.log2(x.astype(np.float64))
    for op in (tac_gpu.HW_LG2, tac_gpu.HW_LG2_FTZ):
        err = np.abs(_run(tac_gpu, op, x) - want)
        assert err.max() <= 2.0**-22, (op, err.max())
    # every binade of normal numbers: the result's roundings grow with its magnitude
    m = _all_floats(1.0, 2.0)[::2048].astype(np.float64)
    xs = (m[None, :] * 2.0 ** np.arange(-125, 127)[:, None]).astype(np.float32).reshape(-1)
    want = np.log2(xs.astype(np.float64))
    for op in (tac_gpu.HW_LG2, tac_gpu.HW_LG2_FTZ):
        err = np.abs(_run(tac_gpu, op, xs) - want)
        assert np.all(err <= 2.0**-22 + 4 * parity.U * np.abs(want)), (op, (err / np.abs(want)).max() / parity.U)
