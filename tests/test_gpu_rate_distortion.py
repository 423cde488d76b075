"""Statistical end-to-end pin of the GPU encode -> decode chain (GB300).

For i.i.d. N(0, 1) rows, y = H D x is again i.i.d. N(0, I) (H and D are
orthogonal), so every pair's angle is uniform on the circle and independent of
its norm (Sec. 2).  With fp32 norms (the angle-only configuration, Sec. 3.1)
the reconstruction error of a pair is r |e^{i delta} - 1| with delta uniform on
[-pi/n, pi/n] (Alg. 1 rounds to the nearest of n bin centres), hence

    E ||x^ - x||^2 / E ||x||^2 = 2 - 2 sin(pi/n) / (pi/n)

exactly.  A wrong bin, a wrong centre, a dropped normalization or a broken
butterfly anywhere in the CUDA path moves the measured ratio off this law.
"""
import math

import pytest

pytestmark = pytest.mark.gpu


def _rel_mse(tac, x, cfg):
    import torch
    cache = tac.encode(x, cfg)
    y = tac.decode(cache, cfg, dtype=torch.float32)
    torch.cuda.synchronize()
    err = (y.double() - x.double()).pow(2).sum()
    return float(err / x.double().pow(2).sum())


@pytest.mark.parametrize("n", [16, 48, 56, 64, 256])
@pytest.mark.parametrize("d", [64, 128])
def test_uniform_angle_distortion_law(tac_gpu, n, d):
    import torch
    g = torch.Generator(device="cuda")
    g.manual_seed(1234 + n + d)
    rows = (1 << 21) // (d // 64)
    x = torch.randn((rows, d), generator=g, device="cuda", dtype=torch.float32)
    cfg = tac_gpu.layer_cfg(d, n, 32, tac_gpu.NORM_FP32, 7, 1, 0)
    got = _rel_mse(tac_gpu, x, cfg)
    a = math.pi / n
    want = 2.0 - 2.0 * math.sin(a) / a
    # 2^21 * 64 / 2 pairs: the estimate's relative standard error is ~2e-4
    assert abs(got / want - 1.0) < 5e-3, (n, d, got, want)


def test_quantized_norms_add_distortion(tac_gpu):
    """Eq. 2 norm quantization can only add error on top of the angle error:
    4-bit log norms > 8-bit linear norms > fp32 norms (relative MSE)."""
    import torch
    g = torch.Generator(device="cuda")
    g.manual_seed(99)
    x = torch.randn((1 << 19, 128), generator=g, device="cuda", dtype=torch.float32)
    m32 = _rel_mse(tac_gpu, x, tac_gpu.layer_cfg(128, 64, 32, tac_gpu.NORM_FP32))
    m8 = _rel_mse(tac_gpu, x, tac_gpu.layer_cfg(128, 64, 8, tac_gpu.NORM_LINEAR))
    m4 = _rel_mse(tac_gpu, x, tac_gpu.layer_cfg(128, 64, 4, tac_gpu.NORM_LOG))
    assert m32 < m8 < m4, (m32, m8, m4)
