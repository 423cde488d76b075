"""Element-by-element comparison of the CUDA path with the CPU oracle.

Rules:

angle codes   bit-exact wherever the oracle's angle lies 1e-5 rad or more from a
              bin edge; inside that band a differing code is counted, and the
              count must not exceed 1e-6 of all codes (below 10^6 codes: zero).
norm codes    the same rule on Eq. 2: bit-exact wherever the oracle's Eq. 2
              value lies more than 1e-4 code units from a rounding midpoint;
              inside, a code may differ by one level, is counted, and the count
              must not exceed 1e-6 of all codes (below 10^6 codes: zero).
              Structured rows (constants, one-hots) get no exemption.
header        the stored (r_min, r_max) are floating-point outputs:
              |r_gpu - r_oracle| <= (2/sqrt d) gamma + (E_SQRT + 2u) r_max,
              gamma = (log2 d - 1) u ||x||_1 the first-order bound of the fp32
              butterfly on a pair (u = 2^-24), 2u the rounding of the pair
              energy and of the stored value, E_SQRT the hardware square root's
              relative error (a GPU test measures it against this bound).
fp32 norms    (mode 2, Sec. 3.1) the same bound with r in place of r_max; there
              is no header.
decode        on identical codes: fp32 out |y - v| <= 1e-5 ||x^||;
              bf16 out |y - v| <= ulp_bf16(v)/2 + 1e-3 ||x^||  (v = oracle fp64 output).
"""
from __future__ import annotations

import math

import numpy as np

U = 2.0**-24
ANGLE_BAND = 1e-5      # rad: angle codes may differ only this close to a bin edge
NORM_BAND = 1e-4       # code units: norm codes may differ only this close to a midpoint
MISMATCH_RATE = 1e-6   # largest share of codes allowed to differ inside a band
E_SQRT = 2.0**-23      # relative error bound of the hardware square root the kernels use


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


def _allowed(codes: int) -> int:
    """Mismatches allowed inside a band: 1e-6 of the codes, rounded down (0 below 10^6)."""
    return int(MISMATCH_RATE * codes)


def compare_encode(orc, x64: np.ndarray, ref: dict, k, c, hdr, n: int, b: int, mode: int,
                   label: str = "") -> dict:
    """Check GPU codes (k, c, hdr) against oracle output `ref` for input rows x64;
    returns the counts (band populations and mismatches)."""
    rows, d = x64.shape
    P = d // 2
    st = {"label": label, "rows": rows, "codes": rows * P}

    # ---- angle codes ----
    mism = k != ref["k"]
    in_band = ref["edge"] < ANGLE_BAND
    outside = mism & ~in_band
    st["angle_mismatch"] = int(mism.sum())
    st["angle_mismatch_outside_band"] = int(outside.sum())
    st["angle_band_population"] = int(in_band.sum())
    assert st["angle_mismatch_outside_band"] == 0, (label, np.argwhere(outside)[:5])
    assert st["angle_mismatch"] <= _allowed(st["codes"]), (label, st)

    gam = _gamma(x64)
    assert np.all(np.isfinite(gam)), (label, "non-finite input row")
    if mode == FP32_MODE:
        # ---- fp32 norms: values, not codes ----
        r = ref["r"]
        rg = np.ascontiguousarray(c, dtype=np.int32).view(np.float32).astype(np.float64)
        eps_r = (2.0 / math.sqrt(d)) * gam[:, None] + (E_SQRT + 2 * U) * r + 1e-45
        err = np.abs(rg - r)
        st["norm_max_err_over_bound"] = float((err / eps_r).max()) if rows else 0.0
        assert np.all(err <= eps_r), (label, st)
        return st

    # ---- header ----
    hmax_o = ref["hdr"][:, 1].astype(np.float64)
    eps_h = (2.0 / math.sqrt(d)) * gam + (E_SQRT + 2 * U) * hmax_o + 1e-45
    dh = np.abs(hdr.astype(np.float64) - ref["hdr"].astype(np.float64))
    st["header_max_err_over_bound"] = float((dh / eps_h[:, None]).max()) if rows else 0.0
    hmax_ulp = np.spacing(np.abs(ref["hdr"]).astype(np.float32)).astype(np.float64)
    st["header_max_err_ulp"] = float((dh / hmax_ulp).max()) if rows else 0.0
    assert np.all(dh <= eps_h[:, None]), (label, st)

    # ---- norm codes ----
    pre = ref["pre"]
    assert np.all(np.isfinite(pre)), (label, "non-finite Eq. 2 value")
    dist_mid = np.abs(pre - (np.floor(pre) + 0.5))  # distance to the nearest rounding midpoint
    in_band = dist_mid <= NORM_BAND
    nm = c != ref["c"]
    bad = nm & ((np.abs(c.astype(np.int64) - ref["c"]) != 1) | ~in_band)
    st["norm_mismatch"] = int(nm.sum())
    st["norm_mismatch_outside_band"] = int(bad.sum())
    st["norm_band_population"] = int(in_band.sum())
    assert st["norm_mismatch_outside_band"] == 0, (label, st, np.argwhere(bad)[:5])
    assert st["norm_mismatch"] <= _allowed(st["codes"]), (label, st)
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
