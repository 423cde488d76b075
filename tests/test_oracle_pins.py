"""Pins of the CPU oracle against what the paper and the mathematics fix.

None of these re-types the oracle's own formula: each checks a property that a
plausible mistake in the oracle (a transposed Hadamard order, a wrong pairing,
a dropped 1/2 in the rounding, a sign error, a wrong norm scale, a swapped
min/max, a packing off by one) would break.
"""
import math
import os

import numpy as np
import pytest
from scipy import stats

import workloads

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _butterfly(x):
    """A test-local in-place Walsh-Hadamard butterfly (unnormalized), independent of the oracle."""
    y = np.array(x, dtype=np.float64, copy=True)
    d = y.shape[-1]
    h = 1
    while h < d:
        y = y.reshape(*y.shape[:-1], d // (2 * h), 2, h)
        a = y[..., 0, :].copy()
        b = y[..., 1, :].copy()
        y[..., 0, :] = a + b
        y[..., 1, :] = a - b
        y = y.reshape(*y.shape[:-3], d)
        h *= 2
    return y


# ---------------------------------------------------------------------------
# D: SplitMix64 signs (reading R8)
# ---------------------------------------------------------------------------
def test_splitmix64_published_outputs(orc):
    rows = [l.split() for l in open(os.path.join(GOLDEN, "splitmix64_seed0.txt")) if l.strip() and not l.startswith("#")]
    for idx, val in rows:
        assert orc.splitmix64(0, int(idx)) == int(val, 16)


def test_signs_balanced_and_distinct(orc):
    d = 128
    seen = set()
    for layer in range(32):
        for kv in (0, 1):
            s = orc.signs(0, layer, kv, d)
            assert set(np.unique(s)) <= {-1, 1}
            neg = int((s < 0).sum())
            # two-sided binomial test of P(s = -1) = 1/2
            assert stats.binomtest(neg, d, 0.5).pvalue > 1e-4
            seen.add(s.tobytes())
    assert len(seen) == 64  # one D per (layer, K/V)
    # shared mode: the paper's single D (Sec. 3.1), identical for every (layer, kv)
    base = orc.signs(0, 0, 0, d, shared=True)
    for layer in (0, 5, 31):
        for kv in (0, 1):
            assert np.array_equal(orc.signs(0, layer, kv, d, shared=True), base)
    # all 2^16 layer/kv/seed combinations over many draws: overall balance
    allneg = sum(int((orc.signs(seed, 0, 0, 64) < 0).sum()) for seed in range(200))
    assert stats.binomtest(allneg, 200 * 64, 0.5).pvalue > 1e-4


def test_sign_bits_are_bit63_of_stream(orc):
    # s_j = -1 iff bit 63 of output j of the stream keyed by output q of the seed stream.
    seed, layer, kv, d = 12345, 3, 1, 64
    key = orc.splitmix64(seed, 2 * layer + kv)
    want = np.array([-1 if (orc.splitmix64(key, j) >> 63) else 1 for j in range(d)], dtype=np.int8)
    assert np.array_equal(orc.signs(seed, layer, kv, d), want)


# ---------------------------------------------------------------------------
# H: normalized Sylvester Hadamard (Sec. 2)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("d", [2, 4, 8, 16, 32, 64, 128])
def test_hadamard_orthonormal_symmetric_involution(orc, d):
    H = orc.hadamard(d)
    assert np.allclose(np.abs(H), 1.0 / math.sqrt(d), rtol=0, atol=1e-15)
    assert np.array_equal(H, H.T)
    assert np.allclose(H @ H, np.eye(d), rtol=0, atol=1e-12)
    e0 = np.zeros(d); e0[0] = 1.0
    assert np.allclose(H @ e0, np.full(d, 1 / math.sqrt(d)), atol=1e-15)
    assert np.allclose(H @ np.ones(d), math.sqrt(d) * e0, atol=1e-12)


@pytest.mark.parametrize("d", [2, 4, 8, 16])
def test_butterfly_equals_dense_bruteforce(orc, d):
    """The O(d log d) butterfly of Sec. 2 equals the dense matrix (Sylvester order):
    every basis vector, and random vectors."""
    H = orc.hadamard(d)
    eye = np.eye(d)
    assert np.allclose(_butterfly(eye) / math.sqrt(d), H, atol=1e-15)
    x = np.random.default_rng(1).standard_normal((50, d))
    ones = np.ones(d, dtype=np.int8)
    assert np.allclose(orc.transform(x, ones), _butterfly(x) / math.sqrt(d), atol=1e-12)


def test_hadamard_d2_d4_explicit(orc):
    s = 1 / math.sqrt(2)
    assert np.allclose(orc.hadamard(2), [[s, s], [s, -s]])
    H4 = 0.5 * np.array([[1, 1, 1, 1], [1, -1, 1, -1], [1, 1, -1, -1], [1, -1, -1, 1]])
    assert np.allclose(orc.hadamard(4), H4)


@pytest.mark.parametrize("d", [16, 64, 128])
def test_transform_preserves_norm_and_applies_D_first(orc, d):
    rng = np.random.default_rng(2)
    x = rng.standard_normal((40, d)) * np.exp(rng.standard_normal(d))
    s = orc.signs(7, 1, 0, d)
    y = orc.transform(x, s)
    assert np.allclose(np.linalg.norm(y, axis=1), np.linalg.norm(x, axis=1), rtol=1e-12)
    # y = H (s * x): applying H again and undoing D returns x (H^-1 = H, D^-1 = D)
    back = orc.transform(y, np.ones(d, dtype=np.int8)) * s
    assert np.allclose(back, x, atol=1e-12 * np.abs(x).max())


# ---------------------------------------------------------------------------
# Angle quantizer (Alg. 1)
# ---------------------------------------------------------------------------
def _x_from_y(orc, y, s):
    """x with H D x = y exactly in exact arithmetic: x = D H y."""
    d = y.shape[1]
    return orc.transform(y, np.ones(d, dtype=np.int8)) * s


@pytest.mark.parametrize("n", [8, 16, 48, 56, 64, 256])
def test_angle_worked_examples(orc, n):
    d = 64  # 1/sqrt(64) = 1/8: x = D H y is exact
    s = orc.signs(3, 0, 0, d)
    pairs = [((1, 0), 0), ((0, 1), n // 4), ((-1, 0), n // 2), ((0, -1), 3 * n // 4), ((1, 1), n // 8),
             ((-1, -1), 5 * n // 8), ((3, 0), 0), ((0, 0.5), n // 4)]
    y = np.zeros((1, d))
    for i, ((a, b), _) in enumerate(pairs):
        y[0, 2 * i], y[0, 2 * i + 1] = a, b
    x = _x_from_y(orc, y, s)
    out = orc.encode(x, s, n, 8, 0)
    for i, (_, k) in enumerate(pairs):
        assert out["k"][0, i] == k, (i, pairs[i], out["k"][0, i])
    # remaining pairs are (0, 0): reading R3 gives bin 0
    assert np.all(out["k"][0, len(pairs):] == 0)


def test_angle_n2_halfplane_and_n4_nearest_axis(orc):
    d = 16
    s = np.ones(d, dtype=np.int8)
    rng = np.random.default_rng(5)
    y = rng.standard_normal((200, d))
    x = _x_from_y(orc, y, s)
    k2 = orc.encode(x, s, 2, 8, 0)["k"]
    k4 = orc.encode(x, s, 4, 8, 0)["k"]
    y0, y1 = y[:, 0::2], y[:, 1::2]
    assert np.array_equal(k2, (y0 < 0).astype(np.int32))          # n = 2: left half-plane
    ang = np.mod(np.arctan2(y1, y0), 2 * np.pi)
    axis = np.argmin(np.abs(np.angle(np.exp(1j * (ang[..., None] - np.arange(4) * np.pi / 2)))), axis=-1)
    assert np.array_equal(k4, axis.astype(np.int32))               # n = 4: nearest axis


@pytest.mark.parametrize("n", [16, 48, 56, 64, 256])
def test_angle_error_bound(orc, n):
    """|theta^ - theta| <= pi/n (wrapped) for every pair, theta^ = 2 pi k / n."""
    d = 128
    w = workloads.CONFIGS["mistral7b"]
    sig = workloads.channel_scales(w, 0, 0)[0]
    x = workloads.scaled_gaussian_rows(300, d, sig, seed=1)
    s = orc.signs(0, 0, 0, d)
    y = orc.transform(x, s)
    out = orc.encode(x, s, n, 8, 0)
    theta = np.arctan2(y[:, 1::2], y[:, 0::2])
    err = np.angle(np.exp(1j * (theta - 2 * np.pi * out["k"] / n)))
    assert np.all(np.abs(err) <= np.pi / n * (1 + 1e-12))
    # edge distance diagnostic is consistent: half a bin minus the error
    assert np.allclose(out["edge"], np.pi / n - np.abs(err), atol=1e-9)


def test_angle_uniform_for_iid_gaussian(orc):
    """Sec. 2: for spherically symmetric pairs the angle is uniform; y = H D x of an
    i.i.d. Gaussian x is exactly N(0, I), so the n bins are equally likely."""
    d, n = 128, 64
    x = workloads.iid_gaussian_rows(2000, d, seed=3)
    s = orc.signs(0, 0, 0, d)
    k = orc.encode(x, s, n, 8, 0)["k"].ravel()
    counts = np.bincount(k, minlength=n)
    assert stats.chisquare(counts).pvalue > 1e-3


def test_angle_density_for_channel_scaled_rows(orc):
    """With channel scales sigma_j, (y_2i, y_2i+1) is a 2-D Gaussian with equal
    variances and correlation rho = sum_j (-1)^j sigma_j^2 / sum_j sigma_j^2 (the
    Sylvester rows 2i and 2i+1 differ exactly by (-1)^j, and D cancels in the
    covariance), so theta has density sqrt(1-rho^2) / (2 pi (1 - rho sin 2 theta)).
    This pins the Hadamard order and the consecutive pairing of Alg. 1."""
    d, n = 128, 32
    rng = np.random.default_rng(11)
    sig = np.exp(rng.normal(0, 1.0, d))
    sig[::2] *= 2.0  # force a strong even/odd energy imbalance: large |rho|
    rho = float(np.sum(((-1.0) ** np.arange(d)) * sig**2) / np.sum(sig**2))
    assert abs(rho) > 0.3
    x = workloads.scaled_gaussian_rows(4000, d, sig, seed=4)
    s = orc.signs(0, 2, 1, d)
    k = orc.encode(x, s, n, 8, 0)["k"].ravel()
    counts = np.bincount(k, minlength=n)
    f = lambda t: math.sqrt(1 - rho * rho) / (2 * math.pi * (1 - rho * math.sin(2 * t)))
    from scipy.integrate import quad
    probs = np.array([quad(f, 2 * math.pi * (j - 0.5) / n, 2 * math.pi * (j + 0.5) / n)[0] for j in range(n)])
    assert abs(probs.sum() - 1) < 1e-9
    assert stats.chisquare(counts, probs * counts.sum()).pvalue > 1e-3
    # and the uniform law is rejected (the effect is real)
    assert stats.chisquare(counts).pvalue < 1e-6


# ---------------------------------------------------------------------------
# Norm quantizer (Sec. 3.3, Eq. 2)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 0), (8, 1), (4, 1)])
def test_norm_endpoints_and_error_bound(orc, b, mode):
    d = 128
    w = workloads.CONFIGS["mistral7b"]
    x = np.asarray(workloads.block(w, 0, mode, tokens=64).float().numpy(), dtype=np.float64)
    s = orc.signs(0, 0, mode, d)
    out = orc.encode(x, s, 64, b, mode)
    L = (1 << b) - 1
    r = out["r"]
    c = out["c"]
    hmin, hmax = out["hdr"][:, 0].astype(np.float64), out["hdr"][:, 1].astype(np.float64)
    # stored min/max are the fp32 roundings of the extreme norms
    assert np.array_equal(out["hdr"][:, 1], r.max(axis=1).astype(np.float32))
    if mode == 0:
        assert np.array_equal(out["hdr"][:, 0], r.min(axis=1).astype(np.float32))
    # argmax pair gets the top code, argmin pair the bottom code
    rows = np.arange(len(r))
    assert np.all(c[rows, r.argmax(axis=1)] == L)
    assert np.all(c[rows, r.argmin(axis=1)] == 0)
    # reconstruction error of the norm within half a step (plus fp32 header slack)
    if mode == 0:
        step = (hmax - hmin) / L
        rhat = hmin[:, None] + c * step[:, None]
        assert np.all(np.abs(rhat - r) <= step[:, None] / 2 + 4e-7 * hmax[:, None])
    else:
        lr = np.log2(np.maximum(r, hmax[:, None] * 2.0**-24))
        lmin, lmax = np.log2(hmin), np.log2(hmax)
        step = (lmax - lmin) / L
        lhat = lmin[:, None] + c * step[:, None]
        assert np.all(np.abs(lhat - lr) <= step[:, None] / 2 + 1e-6)


def test_eq2_takes_the_exact_extremes(orc):
    """Reading R4: Eq. 2 normalizes by the vector's own minimum and maximum norm,
    so the argmax pair's value is exactly 2^b - 1 and the argmin pair's exactly 0
    (against the fp32-rounded header they would be off by ~1e-8 relative).  The
    header still holds the fp32 roundings of both."""
    d = 128
    w = workloads.CONFIGS["mistral7b"]
    x = np.asarray(workloads.block(w, 2, 0, tokens=40).float().numpy(), dtype=np.float64)
    rows = np.arange(len(x))
    for b, mode in ((8, 0), (4, 1), (8, 1)):
        s = orc.signs(0, 2, mode, d)
        out = orc.encode(x, s, 64, b, mode)
        r, pre = out["r"], out["pre"]
        L = (1 << b) - 1
        assert np.all(pre[rows, r.argmax(axis=1)] == L)
        if mode == 0:
            assert np.all(pre[rows, r.argmin(axis=1)] == 0.0)
        assert np.array_equal(out["hdr"][:, 1], r.max(axis=1).astype(np.float32))
        # rows whose extremes are not fp32 numbers exist, so the two readings differ here
        assert np.any(r.max(axis=1) != r.max(axis=1).astype(np.float32).astype(np.float64))


def _pairs_at_axes(orc, norms, n, s):
    """Rows with pair i = norms[i] * (cos, sin)(2 pi k_i / n), k_i on the axes
    (multiples of n/4), so that x = D H y is exact at d = 64 (H = +-1/8)."""
    rows, P = norms.shape
    rng = np.random.default_rng(7)
    q = rng.integers(0, 4, size=(rows, P))
    k = q * (n // 4)
    y = np.zeros((rows, 2 * P))
    y[:, 0::2] = norms * np.array([1.0, 0.0, -1.0, 0.0])[q]
    y[:, 1::2] = norms * np.array([0.0, 1.0, 0.0, -1.0])[q]
    return _x_from_y(orc, y, s), y, k


@pytest.mark.parametrize("b,base", [(4, 0), (4, -10), (3, 5), (2, -3)])
def test_log_dequant_exact_at_powers_of_two(orc, b, base):
    """Sec. 3.3 log-space variant with reading R7: pair norms 2^(base + j),
    j = 0 .. 2^b - 1 (both extremes present), span exactly 2^b - 1 octaves, so
    Eq. 2 on log r gives the integer code j with no rounding, and decode must
    return 2^(base + c) exactly: a wrong log base or exp base, 2^b instead of
    2^b - 1 levels, or swapped l_min / l_max all break it."""
    d, n = 64, 16
    L = (1 << b) - 1
    rng = np.random.default_rng(b * 100 + base)
    j = rng.integers(0, L + 1, size=(12, d // 2))
    j[:, 0], j[:, 1] = 0, L
    s = orc.signs(0, 1, 1, d)
    x, y, k = _pairs_at_axes(orc, 2.0 ** (base + j), n, s)
    out = orc.encode(x, s, n, b, 1)
    assert np.array_equal(out["c"], j.astype(np.int32))
    assert np.array_equal(out["k"], k.astype(np.int32))
    assert np.all(out["hdr"][:, 0] == np.float32(2.0**base)) and np.all(out["hdr"][:, 1] == np.float32(2.0 ** (base + L)))
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, b, 1)
    assert np.allclose(xh, x, rtol=0, atol=1e-12 * np.abs(x).max())


def test_log_dequant_floor(orc):
    """Reading R6: norms below 2^-24 r_max are floored there before the log, and
    the header's r_min is that floor.  With b = 2 and norms 2^0 .. 2^24 in steps
    of 2^8 plus one pair at 2^-5, the floored pair takes code 0 and decodes to
    the floor 2^0, the others decode exactly."""
    d, n = 64, 16
    j = np.tile(np.array([0, 8, 16, 24]), (3, 8)).astype(np.float64)
    norms = 2.0**j
    norms[:, 5] = 2.0**-5
    s = orc.signs(2, 0, 1, d)
    x, y, k = _pairs_at_axes(orc, norms, n, s)
    out = orc.encode(x, s, n, 2, 1)
    want = (j // 8).astype(np.int32)
    want[:, 5] = 0
    assert np.array_equal(out["c"], want)
    assert np.all(out["hdr"][:, 0] == 1.0) and np.all(out["hdr"][:, 1] == np.float32(2.0**24))
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, 2, 1)
    yh = orc.transform(xh, s)
    rh = np.hypot(yh[:, 0::2], yh[:, 1::2])
    expect = norms.copy()
    expect[:, 5] = 1.0
    # the re-transform rounds at the scale of the largest pair (2^24)
    assert np.allclose(rh, expect, rtol=1e-12, atol=1e-12 * 2.0**24)


@pytest.mark.parametrize("b", [4, 8])
def test_log_dequant_half_step(orc, b):
    """Decoded norms in log-space mode lie within half a log step of log2 r
    (floored at 2^-24 r_max): |log2 r^ - log2 r| <= (l_max - l_min) / (2 (2^b - 1)),
    up to the fp32 rounding of the stored header.  r^ is measured on the decoded
    vector itself (y^ = H D x^), not recomputed from the codes."""
    d, n = 128, 64
    w = workloads.CONFIGS["mistral7b"]
    x = np.asarray(workloads.block(w, 7, 1, tokens=48).float().numpy(), dtype=np.float64)
    s = orc.signs(0, 7, 1, d)
    out = orc.encode(x, s, n, b, 1)
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, b, 1)
    yh = orc.transform(xh, s)
    rh = np.hypot(yh[:, 0::2], yh[:, 1::2])
    r = np.maximum(out["r"], out["r"].max(axis=1, keepdims=True) * 2.0**-24)
    hmin, hmax = out["hdr"][:, 0].astype(np.float64), out["hdr"][:, 1].astype(np.float64)
    half = (np.log2(hmax) - np.log2(hmin)) / (2 * ((1 << b) - 1))
    err = np.abs(np.log2(rh) - np.log2(r))
    assert np.all(err <= half[:, None] + 2e-7), float((err - half[:, None]).max())
    assert np.all(rh >= hmin[:, None] * (1 - 1e-12)) and np.all(rh <= hmax[:, None] * (1 + 1e-12))
    # the bound is attained up to a small factor (the test would catch a zero step)
    assert float((err / half[:, None]).max()) > 0.9


def test_norm_monotone(orc):
    d = 64
    rng = np.random.default_rng(9)
    x = rng.standard_normal((100, d))
    s = orc.signs(1, 0, 0, d)
    out = orc.encode(x, s, 16, 8, 0)
    for row in range(100):
        order = np.argsort(out["r"][row], kind="stable")
        assert np.all(np.diff(out["c"][row][order]) >= 0)


def test_degenerate_rows(orc):
    d = 64
    s = orc.signs(0, 0, 0, d)
    zero = np.zeros((3, d))
    for mode in (0, 1):
        out = orc.encode(zero, s, 64, 8, mode)
        assert np.all(out["k"] == 0) and np.all(out["c"] == 0) and np.all(out["hdr"] == 0)
        y = orc.decode(out["k"], out["c"], out["hdr"], s, 64, 8, mode)
        assert np.all(y == 0)
    # every pair norm equal: r_max == r_min -> all norm codes 0, decode keeps r
    y = np.zeros((1, d))
    y[0, 0::2] = 1.0   # every pair (1, 0): equal norms, angle 0
    x = _x_from_y(orc, y, s)
    out = orc.encode(x, s, 64, 4, 1)
    assert np.all(out["c"] == 0)
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, 64, 4, 1)
    assert np.allclose(xh, x, atol=1e-6)


# ---------------------------------------------------------------------------
# Decode (Sec. 3.1) and whole round trips
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("n", [8, 48, 56, 64, 256])
def test_exact_round_trip_at_bin_centres(orc, n):
    """y with every angle on a bin centre and norms in {1, 2}: encode gives the
    known codes and decode returns x (1-bit linear norms are exact here)."""
    d = 64
    rng = np.random.default_rng(n)
    k = rng.integers(0, n, size=(20, d // 2))
    r = rng.integers(1, 3, size=(20, d // 2)).astype(np.float64)
    r[:, 0], r[:, 1] = 1.0, 2.0  # both levels present in every row
    y = np.zeros((20, d))
    y[:, 0::2] = r * np.cos(2 * np.pi * k / n)
    y[:, 1::2] = r * np.sin(2 * np.pi * k / n)
    s = orc.signs(0, 4, 1, d)
    x = _x_from_y(orc, y, s)
    # norm bits: the oracle's Eq. 2 at b = 4 maps {1, 2} to codes {0, 15}
    out = orc.encode(x, s, n, 4, 0)
    assert np.array_equal(out["k"], k.astype(np.int32))
    assert np.array_equal(out["c"], np.where(r > 1.5, 15, 0).astype(np.int32))
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, 4, 0)
    assert np.allclose(xh, x, atol=1e-12)


@pytest.mark.parametrize("n", [16, 56, 64, 256])
def test_decode_pair_error_bound(orc, n):
    """With (nearly) unquantized norms the reconstruction error of each pair is
    at most the chord of half a bin, 2 r sin(pi / 2n), and H is orthonormal so
    ||x^ - x||^2 is the sum of the pair errors."""
    d = 128
    rng = np.random.default_rng(21)
    x = rng.standard_normal((50, d)) * np.exp(rng.normal(0, 1, d))
    s = orc.signs(0, 0, 0, d)
    out = orc.encode(x, s, n, 16, 0)   # 16-bit linear norms: norm error ~1e-5 of the range
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, 16, 0)
    r = out["r"]
    hmin, hmax = out["hdr"][:, 0].astype(np.float64), out["hdr"][:, 1].astype(np.float64)
    norm_err = (hmax - hmin) / 65535 / 2 + 1e-7 * hmax
    bound = np.sqrt(np.sum((2 * r * math.sin(math.pi / (2 * n)) + norm_err[:, None]) ** 2, axis=1))
    assert np.all(np.linalg.norm(xh - x, axis=1) <= bound * (1 + 1e-9) + 1e-12)


# ---------------------------------------------------------------------------
# fp32 norm storage (reading R16: the angle-only configuration of Sec. 3.1 and
# Tables 1-4, "each pair norm r_i is stored in fp32")
# ---------------------------------------------------------------------------
def test_fp32_norms_store_exact_norms(orc):
    """Pairs built from scaled Pythagorean triples have exactly representable
    norms (3-4-5, 5-12-13, 8-15-17); x = D H y is exact at d = 64.  The stored
    norm code is the fp32 bit pattern of that norm, and decode equals an
    independent reconstruction D H y^ (test-local butterfly) from the stored
    norm and the bin-centre angle."""
    d, n = 64, 56
    triples = [(3, 4, 5), (5, 12, 13), (8, 15, 17), (-3, 4, 5), (4, -3, 5), (-12, -5, 13)]
    rng = np.random.default_rng(2)
    y = np.zeros((8, d))
    rr = np.zeros((8, d // 2))
    for row in range(8):
        for i in range(d // 2):
            a, b, c = triples[rng.integers(len(triples))]
            sc = 2.0 ** int(rng.integers(-4, 4))
            y[row, 2 * i], y[row, 2 * i + 1], rr[row, i] = a * sc, b * sc, c * sc
    s = orc.signs(1, 2, 1, d)
    x = _x_from_y(orc, y, s)
    out = orc.encode(x, s, n, 32, 2)
    assert np.array_equal(out["c"].view(np.float32).astype(np.float64), rr)
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, 32, 2)
    phi = 2 * np.pi * out["k"] / n
    yh = np.zeros((8, d))
    yh[:, 0::2], yh[:, 1::2] = rr * np.cos(phi), rr * np.sin(phi)
    want = _butterfly(yh) / math.sqrt(d) * s
    assert np.allclose(xh, want, rtol=0, atol=1e-12 * np.abs(want).max())


@pytest.mark.parametrize("n", [48, 64, 256])
def test_fp32_norms_pair_error_bound(orc, n):
    """fp32 norms: each pair's reconstruction error is at most the chord of half
    a bin, 2 r sin(pi/2n), plus the fp32 rounding of r (2^-24 r)."""
    d = 128
    rng = np.random.default_rng(30 + n)
    x = rng.standard_normal((40, d)) * np.exp(rng.normal(0, 1, d))
    s = orc.signs(0, 5, 0, d)
    out = orc.encode(x, s, n, 32, 2)
    xh = orc.decode(out["k"], out["c"], out["hdr"], s, n, 32, 2)
    r = out["r"]
    bound = np.sqrt(np.sum((2 * r * math.sin(math.pi / (2 * n)) + r * 2.0**-24) ** 2, axis=1))
    assert np.all(np.linalg.norm(xh - x, axis=1) <= bound * (1 + 1e-9) + 1e-12)
    # 16 bits per element: one fp32 per pair (Sec. 3.1)
    assert orc.pack(out["c"][:1], 32).nbytes * 8 / d == 16


# ---------------------------------------------------------------------------
# Packing (reading R9) and rates (Eq. 1, Eq. 3)
# ---------------------------------------------------------------------------
def test_pack_layout_by_hand(orc):
    # codes 1, 2, 3 at 3 bits, LSB-first: bits 001 | 010 | 011 -> 0b11010001, 0b00000000
    out = orc.pack(np.array([[1, 2, 3]]), 3)
    assert out.tolist() == [[0xD1, 0x00]]
    out = orc.pack(np.array([[0xAB, 0x01]]), 8)
    assert out.tolist() == [[0xAB, 0x01]]
    out = orc.pack(np.array([[0x3, 0xC]]), 4)
    assert out.tolist() == [[0xC3]]


@pytest.mark.parametrize("bits", [1, 3, 4, 5, 6, 7, 8, 32])
def test_pack_round_trip(orc, bits):
    rng = np.random.default_rng(bits)
    codes = rng.integers(-(1 << 31), 1 << 31, size=(17, 64)) if bits == 32 else rng.integers(0, 1 << bits, size=(17, 64))
    assert np.array_equal(orc.unpack(orc.pack(codes, bits), 64, bits), codes)


def _parse_rates():
    rows = []
    for line in open(os.path.join(GOLDEN, "rates.txt")):
        if not line.strip() or line.startswith("#"):
            continue
        kind, params, value, where = [f.strip() for f in line.split("|")]
        rows.append((kind, dict(p.split("=") for p in params.split() if "=" in p), float(value), where))
    return rows


def _layers(spec: str, L: int):
    out = set()
    for part in spec.split(","):
        if not part:
            continue
        a, _, b = part.partition("-")
        out.update(range(int(a), int(b or a) + 1))
    return out


def schedule_from_golden(kind, p):
    if kind == "uniform":
        n = int(p["n"])
        return [n], [n]
    L = int(p["L"])
    if kind == "kv":
        return [int(p["nK"])] * L, [int(p["nV"])] * L
    ek, ev = (int(v) for v in p["early"].split(","))
    boosted = _layers(p["layers"], L)
    return ([ek if l in boosted else 128 for l in range(L)], [ev if l in boosted else 64 for l in range(L)])


@pytest.mark.parametrize("row", _parse_rates(), ids=lambda r: f"{r[0]}-{r[3]}-{r[2]}")
def test_printed_rates(orc, row):
    kind, p, value, _ = row
    if kind == "total":
        got = orc.total_bits(float(p["b_angle"]), float(p["b_norm"]), int(p["d"]))
        assert abs(got - value) < 1e-12
    else:
        nk, nv = schedule_from_golden(kind, p)
        got = orc.avg_angle_bits(nk, nv)
        assert abs(got - value) <= 0.005 + 1e-9, (got, value)


def test_payload_bits_formula(orc):
    """Payload bits per element = log2(n)/2 + b/2 (one angle and one norm per pair);
    Eq. 3 adds 64/d for the fp32 min/max."""
    for n in (16, 32, 64, 128, 256):
        for b in (4, 8):
            d = 128
            codes = np.zeros((1, d // 2), dtype=np.int32)
            ang = orc.pack(codes, int(math.log2(n))).nbytes * 8
            nrm = orc.pack(codes, b).nbytes * 8
            assert (ang + nrm) / d == math.log2(n) / 2 + b / 2
            assert (ang + nrm + 64) / d == orc.total_bits(math.log2(n) / 2, b, d)


# ---------------------------------------------------------------------------
# Attention over decoded vectors (the consumer of the Sec. 3.1 reconstruction)
# ---------------------------------------------------------------------------
def test_attend_special_cases(orc):
    rng = np.random.default_rng(40)
    d = 64
    k = rng.standard_normal((5, d))
    v = rng.standard_normal((5, d))
    q = rng.standard_normal((3, d))
    # one token: every query returns it
    assert np.allclose(orc.attend(q, k[:1], v[:1], 0.3), np.repeat(v[:1], 3, axis=0), atol=1e-14)
    # q = 0: uniform weights, the mean of the values
    assert np.allclose(orc.attend(np.zeros((1, d)), k, v, 1.0), v.mean(axis=0, keepdims=True), atol=1e-14)
    # two tokens: weights sigmoid(delta), delta the score difference (closed form)
    qq = np.zeros((1, d)); qq[0, 3] = 1.0
    kk = np.zeros((2, d)); kk[0, 3], kk[1, 3] = 2.0, -0.5
    w0 = 1.0 / (1.0 + math.exp(-(0.7 * 2.0 - 0.7 * -0.5)))
    assert np.allclose(orc.attend(qq, kk, v[:2], 0.7), w0 * v[0] + (1 - w0) * v[1], atol=1e-14)
    # hard limit: a large scale selects the value of the highest score
    s = q @ k.T
    got = orc.attend(q, k, v, 1e4)
    assert np.allclose(got, v[np.argmax(s, axis=1)], atol=1e-9)


def test_attend_rotated_domain_identity(orc):
    """q . (D H y) = (H D q) . y for every y: scores can be taken against the
    rotated query without transforming each decoded row back."""
    d = 128
    rng = np.random.default_rng(41)
    s = orc.signs(5, 3, 0, d)
    q = rng.standard_normal((4, d))
    y = rng.standard_normal((50, d))
    khat = orc.transform(y, np.ones(d, dtype=np.int8)) * s      # D H y (H symmetric)
    qr = orc.transform(q, s)                                     # H D q
    assert np.allclose(q @ khat.T, qr @ y.T, atol=1e-11)


def test_record_slot_order(orc):
    """Reading R9's record order: slot v holds pair phi_d(v).  A bijection of the
    d/2 pairs; the natural order for d <= 32; for d = 64, 128 (L = d/16) the
    slots l + L m (m = 0..3 and 4..7) hold the runs of 4 consecutive pairs
    starting at 4 l and 4 L + 4 l; values written out by hand for d = 128."""
    for d in (2, 4, 8, 16, 32, 64, 128):
        phi = orc.slot_order(d)
        assert sorted(phi.tolist()) == list(range(d // 2)), d
        if d <= 32:
            assert phi.tolist() == list(range(d // 2))
    phi = orc.slot_order(128)
    assert phi[:10].tolist() == [0, 4, 8, 12, 16, 20, 24, 28, 1, 5]
    assert phi[31] == 31 and phi[32] == 32 and phi[33] == 36 and phi[63] == 63
    assert orc.slot_order(64)[:6].tolist() == [0, 4, 8, 12, 1, 5]
    for d in (64, 128):
        L = d // 16
        phi = orc.slot_order(d)
        for l in range(L):
            for h in (0, 1):
                run = sorted(phi[l + L * m] for m in range(4 * h, 4 * h + 4))
                assert run == [4 * L * h + 4 * l + j for j in range(4)], (d, l, h)


def test_record_pack_is_pack_in_slot_order(orc):
    """pack_record = pack of the codes taken in slot order; unpack_record inverts it."""
    rng = np.random.default_rng(5)
    for d in (16, 64, 128):
        for bits in (3, 6, 8, 32):
            codes = rng.integers(0, 2**min(bits, 31), size=(5, d // 2))
            phi = orc.slot_order(d)
            rec = orc.pack_record(codes, d, bits)
            assert np.array_equal(rec, orc.pack(codes[:, phi], bits))
            assert np.array_equal(orc.unpack_record(rec, d, bits), codes)
