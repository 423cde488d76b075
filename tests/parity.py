"""Element-by-element comparison of the CUDA path with the CPU oracle.

Rules (derived in the design notes from the fp32 arithmetic of the kernels):

angle codes   bit-exact wherever the oracle's angle lies 1e-5 rad or more from a
              bin edge; inside that band a differing code is counted, and the
              count must not exceed 1e-6 of all codes (below 10^6 codes: zero).
header        |r_gpu - r_oracle| <= eps_h, eps_h = (2/sqrt d) gamma + 4 u r_max,
              gamma = (log2 d - 1) u ||x||_1: the first-order bound of the fp32
              butterfly's rounding on a pair (u = 2^-24), plus the energy's
              rounding and the hardware square root (<= 2 ulp).
norm codes    bit-exact wherever the oracle's Eq. 2 pre-round value lies more than
              beta_i from a rounding midpoint, beta_i the propagated bound of the
              fp32 norm, header and Eq. 2 arithmetic; inside, a code may differ by
              one level and is counted (rate reported, must stay <= 1e-4).
fp32 norms    (mode 2, Sec. 3.1) |r_gpu - r| <= (2/sqrt d) gamma + 4 u r, r the oracle's
              exact pair norm; there is no header.
decode        on identical codes: fp32 out |y - v| <= 1e-5 ||x^||;
              bf16 out |y - v| <= ulp_bf16(v)/2 + 1e-3 ||x^||  (v = oracle fp64 output).
"""
from __future__ import annotations

import math

import numpy as np

U = 2.0**-24
ANGLE_BAND = 1e-5


def to_f64(t) -> np.ndarray:
    """Exact fp64 copy of a bf16/fp32 torch tensor."""
    import torch
    return t.detach().to("cpu").to(torch.float64).numpy() if t.dtype != torch.float64 else t.cpu().numpy()


def signs_pm1(words: np.ndarray, d: int) -> np.ndarray:
    return np.array([-1 if (int(words[j // 32]) >> (j % 32)) & 1 else 1 for j in range(d)], dtype=np.int8)


def code_bits(n: int) -> int:
    """Bits of one angle code: ceil(log2 n)."""
    return int(math.ceil(math.log2(n)))


FP32_MODE = 2


def gpu_codes(orc, cache, rows: int | None = None, slots: np.ndarray | None = None):
    """(k, c, hdr) read back from a device cache (optionally only some slots).
    With fp32 norms c holds the norms' fp32 bit patterns and hdr is None."""
    cfg = cache.cfg
    codes, norms, hdr = cache.planes()
    sel = slots if slots is not None else (slice(0, rows) if rows is not None else slice(None))
    codes, norms = codes[sel], norms[sel]
    if hdr is not None:
        hdr = np.array(hdr[sel], dtype=np.float32)
    k = orc.unpack_record(codes, cfg.d, code_bits(cfg.n_angle))
    c = orc.unpack_record(norms, cfg.d, cfg.norm_bits)
    return k, c, hdr


def _gamma(x64: np.ndarray) -> np.ndarray:
    d = x64.shape[1]
    return (math.log2(d) - 1) * U * np.abs(x64).sum(axis=1)


def compare_encode(orc, x64: np.ndarray, ref: dict, k, c, hdr, n: int, b: int, mode: int,
                   label: str = "", structured: bool = False) -> dict:
    """Check GPU codes (k, c, hdr) against oracle output `ref` for input rows x64.

    `structured`: hand-built rows (constants, one-hots) put Eq. 2 values exactly on
    rounding midpoints, so only the band rule (not the statistical rate) applies."""
    rows, d = x64.shape
    P = d // 2
    L = (1 << b) - 1
    st = {"label": label, "rows": rows, "codes": rows * P}

    # ---- angle codes ----
    mism = k != ref["k"]
    outside = mism & (ref["edge"] >= ANGLE_BAND)
    st["angle_mismatch"] = int(mism.sum())
    st["angle_mismatch_outside_band"] = int(outside.sum())
    st["angle_band_population"] = int((ref["edge"] < ANGLE_BAND).sum())
    assert st["angle_mismatch_outside_band"] == 0, (label, np.argwhere(outside)[:5])
    assert st["angle_mismatch"] <= 1e-6 * st["codes"], (label, st)

    gam = _gamma(x64)
    if mode == FP32_MODE:
        # ---- fp32 norms: values, not codes ----
        r = ref["r"]
        rg = np.ascontiguousarray(c, dtype=np.int32).view(np.float32).astype(np.float64)
        eps_r = (2.0 / math.sqrt(d)) * gam[:, None] + 4 * U * r + 1e-45
        err = np.abs(rg - r)
        st["norm_max_err_over_bound"] = float((err / eps_r).max()) if rows else 0.0
        assert np.all(err <= eps_r), (label, st)
        return st

    # ---- header ----
    hmax_o = ref["hdr"][:, 1].astype(np.float64)
    eps_h = (2.0 / math.sqrt(d)) * gam + 4 * U * hmax_o + 1e-45
    dh = np.abs(hdr.astype(np.float64) - ref["hdr"].astype(np.float64))
    st["header_max_err_over_bound"] = float((dh / eps_h[:, None]).max()) if rows else 0.0
    assert np.all(dh <= eps_h[:, None]), (label, st)

    # ---- norm codes ----
    hmin_o = ref["hdr"][:, 0].astype(np.float64)
    r = ref["r"]
    eps_r = (2.0 / math.sqrt(d)) * gam[:, None] + 4 * U * r
    dh_range = np.maximum(hmax_o - hmin_o, 1e-300)
    if mode == 0:
        beta = L * (eps_r + 3 * eps_h[:, None]) / dh_range[:, None] + 4 * U * L
    else:
        floor_r = np.maximum(r, hmax_o[:, None] * 2.0**-24)
        lmin = np.log2(np.maximum(hmin_o, 1e-300))
        lmax = np.log2(np.maximum(hmax_o, 1e-300))
        lrange = np.maximum(lmax - lmin, 1e-300)
        # hardware log2: absolute error <= 2^-21 (plus relative rounding of the result)
        dl = (eps_r / floor_r + 2 * U) / math.log(2) + 4 * U * np.abs(np.log2(floor_r)) + 2.0**-21
        dlmin = (eps_h / np.maximum(hmin_o, 1e-300) + 2 * U) / math.log(2) + 4 * U * np.abs(lmin) + 2.0**-21
        dlmax = (eps_h / np.maximum(hmax_o, 1e-300) + 2 * U) / math.log(2) + 4 * U * np.abs(lmax) + 2.0**-21
        beta = L * (dl + 3 * np.maximum(dlmin, dlmax)[:, None]) / lrange[:, None] + 4 * U * L
    flat = (ref["hdr"][:, 0] == ref["hdr"][:, 1])
    beta[flat] = 0.0
    pre = ref["pre"]
    dist_mid = np.abs(pre - (np.floor(pre) + 0.5))  # distance to the nearest rounding midpoint
    nm = c != ref["c"]
    st["norm_mismatch"] = int(nm.sum())
    bad = nm & ((np.abs(c - ref["c"]) != 1) | (dist_mid > beta))
    st["norm_mismatch_outside_band"] = int(bad.sum())
    st["norm_band_population"] = int((dist_mid <= beta).sum())
    assert st["norm_mismatch_outside_band"] == 0, (label, st, np.argwhere(bad)[:5])
    if not structured:
        assert st["norm_mismatch"] <= max(2, 1e-4 * st["codes"]), (label, st)
    return st


def bf16_half_ulp(v: np.ndarray) -> np.ndarray:
    a = np.abs(v)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    return np.where(a > 0, 2.0 ** (e - 8), 2.0**-134)


def compare_decode(y_gpu: np.ndarray, v: np.ndarray, out_dtype: str, label: str = "") -> dict:
    """Decoded rows vs the oracle's fp64 decode of the same codes."""
    nrm = np.linalg.norm(v, axis=1)
    err = np.abs(y_gpu - v)
    if out_dtype == "fp32":
        lim = 1e-5 * nrm[:, None]
    else:
        lim = bf16_half_ulp(v) + 1e-3 * nrm[:, None]
    st = {"label": label, "max_err_over_norm": float((err.max(axis=1) / np.maximum(nrm, 1e-300)).max()) if len(v) else 0.0,
          "max_err_over_limit": float((err / np.maximum(lim, 1e-300)).max()) if len(v) else 0.0}
    assert np.all(err <= lim), (label, st)
    return st
