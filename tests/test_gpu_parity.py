"""CUDA encode/decode vs the CPU oracle, element by element (GB300)."""
import math

import numpy as np
import pytest

import parity
import workloads

pytestmark = pytest.mark.gpu


def _torch():
    import torch
    return torch


def _oracle_cache(tac, orc, cfg, ref):
    """A device cache holding the oracle's own records (for decode on identical codes)."""
    torch = _torch()
    rows = ref["k"].shape[0]
    w = parity.code_bits(cfg.n_angle)
    cache = tac.Cache.empty(cfg, rows)
    ang = orc.pack_record(ref["k"], cfg.d, w).reshape(-1)
    nrm = orc.pack_record(ref["c"], cfg.d, cfg.norm_bits).reshape(-1)
    off = tac.header_offset(cfg, rows)
    nb = np.zeros(tac.norms_bytes(cfg, rows), dtype=np.uint8)
    nb[: nrm.size] = nrm
    if cfg.norm_mode != tac.NORM_FP32:
        nb[off: off + 8 * rows] = ref["hdr"].astype(np.float32).view(np.uint8).reshape(-1)
    if ang.size:
        cache.codes[: ang.size].copy_(torch.from_numpy(ang))
    if nb.size:
        cache.norms[: nb.size].copy_(torch.from_numpy(nb))
    return cache


def check_roundtrip(tac, orc, x, d, n, b, mode, seed=0, layer=0, kv=0, label="", decode_dtypes=("bf16", "fp32")):
    torch = _torch()
    rows = x.shape[0]
    cfg = tac.layer_cfg(d, n, b, mode, seed, layer, kv)
    cache = tac.encode(x, cfg)
    torch.cuda.synchronize()
    x64 = parity.to_f64(x)
    s = orc.signs(seed, layer, kv, d)
    assert np.array_equal(s, parity.signs_pm1(cfg.signs, d))
    ref = orc.encode(x64, s, n, b, mode)
    k, c, hdr = parity.gpu_codes(orc, cache, rows)
    st = parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=label)
    # decode on identical codes (the oracle's records) into bf16 and fp32
    oc = _oracle_cache(tac, orc, cfg, ref)
    v = orc.decode(ref["k"], ref["c"], ref["hdr"], s, n, b, mode)
    for dt in decode_dtypes:
        y = tac.decode(oc, cfg, dtype=torch.bfloat16 if dt == "bf16" else torch.float32)
        torch.cuda.synchronize()
        parity.compare_decode(parity.to_f64(y), v, dt, label=f"{label} decode {dt}")
    # end to end: GPU encode -> GPU decode equals the oracle decode of the GPU's codes
    y2 = tac.decode(cache, cfg, dtype=torch.float32)
    torch.cuda.synchronize()
    v2 = orc.decode(k, c, hdr if hdr is not None else ref["hdr"], s, n, b, mode)
    parity.compare_decode(parity.to_f64(y2), v2, "fp32", label=f"{label} e2e")
    return st


def _rows(w, rows, seed, dtype=None, layer=0, kv=0):
    torch = _torch()
    T = -(-rows // w.heads)
    x = workloads.block(w, layer, kv, tokens=T, seed=seed, device="cuda", dtype=dtype)
    return x[:rows].contiguous()


def test_tiny_config_full(tac_gpu, orc):
    """Config 1: K, V fp32 [8, 1024, 64], n = 64, K 8-bit linear, V 4-bit log, every row."""
    w = workloads.CONFIGS["tiny"]
    for kv in (workloads.K, workloads.V):
        x = workloads.block(w, 0, kv, device="cuda")
        d, n, b, mode = w.codebook(0, kv)
        check_roundtrip(tac_gpu, orc, x, d, n, b, mode, layer=0, kv=kv, label=f"tiny kv={kv}")


@pytest.mark.parametrize("n", [2, 4, 8, 16, 32, 64, 128, 256])
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 1)])
def test_d128_bf16_every_codebook(tac_gpu, orc, n, b, mode):
    w = workloads.CONFIGS["mistral7b"]
    x = _rows(w, 1000, seed=n * 7 + b, layer=n % 32, kv=mode)  # 1000 rows: 7 full tiles + a ragged one
    check_roundtrip(tac_gpu, orc, x, 128, n, b, mode, layer=n % 32, kv=mode, label=f"d128 n={n} b={b}")


@pytest.mark.parametrize("d", [16, 32, 64])
@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 1), (8, 1), (4, 0)])
def test_small_d_and_dtypes(tac_gpu, orc, d, dt, b, mode):
    torch = _torch()
    w = workloads.CONFIGS["llama1b"]
    x = workloads.block(w, 1, 0, tokens=40, seed=d + b, device="cuda")[:, :d] if d <= 64 else None
    x = x.to(torch.bfloat16 if dt == "bf16" else torch.float32).contiguous()
    for n in (16, 256):
        check_roundtrip(tac_gpu, orc, x, d, n, b, mode, seed=3, layer=2, kv=1, label=f"d{d} {dt} n{n}")


@pytest.mark.parametrize("n", [48, 56])
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 1), (32, 2)])
def test_non_power_of_two_bins(tac_gpu, orc, n, b, mode):
    """n = 48, 56 (Table 1): 6-bit codes, bins wrap at n."""
    w = workloads.CONFIGS["mistral7b"]
    x = _rows(w, 777, seed=n + b, layer=5, kv=mode % 2)
    check_roundtrip(tac_gpu, orc, x, 128, n, b, mode, layer=5, kv=mode % 2, label=f"n={n} b={b} m={mode}")
    wl = workloads.CONFIGS["llama1b"]
    x = workloads.block(wl, 2, 1, tokens=60, seed=n, device="cuda")
    check_roundtrip(tac_gpu, orc, x, 64, n, b, mode, seed=1, layer=2, kv=1, label=f"d64 n={n} b={b} m={mode}")


@pytest.mark.parametrize("d", [16, 32, 64, 128])
@pytest.mark.parametrize("dt", ["bf16", "fp32"])
def test_fp32_norms(tac_gpu, orc, d, dt):
    """fp32 pair norms (Sec. 3.1, the angle-only configuration of Tables 1-4)."""
    torch = _torch()
    w = workloads.CONFIGS["mistral7b" if d == 128 else "llama1b"]
    x = workloads.block(w, 3, 0, tokens=50, seed=d, device="cuda")[:, :d]
    x = x.to(torch.bfloat16 if dt == "bf16" else torch.float32).contiguous()
    for n in (2, 64, 256, 56):
        check_roundtrip(tac_gpu, orc, x, d, n, 32, 2, seed=4, layer=3, kv=0, label=f"fp32 norms d{d} {dt} n{n}")


def test_d128_fp32_input(tac_gpu, orc):
    torch = _torch()
    w = workloads.CONFIGS["mistral7b"]
    x = _rows(w, 300, seed=5, dtype=torch.float32)
    check_roundtrip(tac_gpu, orc, x, 128, 64, 8, 0, label="d128 fp32")


@pytest.mark.parametrize("rows", [0, 1, 31, 127, 128, 129, 255, 257])
def test_ragged_row_counts(tac_gpu, orc, rows):
    w = workloads.CONFIGS["mistral7b"]
    torch = _torch()
    if rows == 0:
        cfg = tac_gpu.layer_cfg(128, 64, 8, 0)
        x = torch.empty((0, 128), dtype=torch.bfloat16, device="cuda")
        cache = tac_gpu.encode(x, cfg)
        y = tac_gpu.decode(cache, cfg, rows=0)
        assert y.shape == (0, 128)
        return
    x = _rows(w, rows, seed=rows)
    check_roundtrip(tac_gpu, orc, x, 128, 256, 8, 0, label=f"rows={rows}")
    check_roundtrip(tac_gpu, orc, x, 128, 64, 4, 1, kv=1, label=f"rows={rows} V")


def test_strided_rows(tac_gpu, orc):
    """Rows that are not contiguous (row_stride > d), e.g. one head of a [T, H, d] cache."""
    torch = _torch()
    w = workloads.CONFIGS["mistral7b"]
    big = _rows(w, 600, seed=9).reshape(200, 3, 128)
    x = big[:, 1, :]
    assert x.stride(0) == 384
    check_roundtrip(tac_gpu, orc, x, 128, 64, 8, 0, label="strided")


def test_degenerate_rows(tac_gpu, orc):
    """Zero rows, constant rows, one-hot rows, huge and tiny magnitudes."""
    torch = _torch()
    d = 128
    rng = np.random.default_rng(0)
    rows = [np.zeros(d), np.ones(d), np.full(d, -3.0)]
    for j in (0, 1, 64, 127):
        e = np.zeros(d); e[j] = 2.5
        rows.append(e)
    rows.append(rng.standard_normal(d) * 2.0**50)
    rows.append(rng.standard_normal(d) * 2.0**-60)
    a = np.zeros(d); a[::2] = 1.0          # only even elements
    rows.append(a)
    a = np.zeros(d); a[1::2] = -1.0        # only odd elements
    rows.append(a)
    x = torch.tensor(np.array(rows), dtype=torch.float32).to(torch.bfloat16).cuda()
    for n, b, mode in ((64, 8, 0), (64, 4, 1), (4, 8, 0), (2, 4, 1), (256, 8, 1)):
        check_roundtrip(tac_gpu, orc, x, d, n, b, mode, label=f"degenerate n={n} b={b} m={mode}")


def test_exact_bin_centres_and_ties(tac_gpu, orc):
    """Pairs built on bin centres (robust codes) and on the n = 4 edges at pi/4
    multiples where the oracle's rounding is exact (ties round up)."""
    torch = _torch()
    d = 64
    s = orc.signs(0, 0, 0, d)
    y = np.zeros((4, d))
    y[0, 0::2], y[0, 1::2] = 1.0, 1.0        # theta = pi/4: n = 4 edge, tie -> k = 1
    y[1, 0::2], y[1, 1::2] = 2.0, 0.0        # theta = 0
    y[2, 0::2], y[2, 1::2] = 0.0, 3.0        # theta = pi/2
    y[3, 0::2], y[3, 1::2] = -1.0, 0.0       # theta = pi
    x = orc.transform(y, np.ones(d, dtype=np.int8)) * s   # x = D H y, exact (1/sqrt(64) = 1/8)
    xt = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).cuda()
    assert np.array_equal(parity.to_f64(xt), x)
    for n in (4, 8, 64, 256):
        cfg = tac_gpu.layer_cfg(d, n, 8, 0, 0, 0, 0)
        cache = tac_gpu.encode(xt, cfg)
        torch.cuda.synchronize()
        k, c, hdr = parity.gpu_codes(orc, cache, 4)
        want = orc.encode(x, s, n, 8, 0)["k"]
        assert np.array_equal(k, want), (n, k[:, :3], want[:, :3])
        if n == 4:
            assert np.all(k[0] == 1) and np.all(k[1] == 0) and np.all(k[2] == 1) and np.all(k[3] == 2)


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 1)])
def test_magnitude_range_limits(tac_gpu, orc, dt, b, mode):
    """Rows at the ends of the documented input range, every nonzero |x_j| in
    [2^-53, 2^56] (bf16) or [2^-37, 2^56] (fp32), where every nonzero pair
    energy E^2 + O^2 is a normal fp32 number: rows of the smallest values, rows
    of the largest (whose energy sum overflows, so every pair takes the exact
    path) and rows spread over the whole range with zeros."""
    torch = _torch()
    d = 128
    lo = -53 if dt == "bf16" else -37
    rng = np.random.default_rng(7 + b + 2 * mode)

    def row(elo, ehi, zero_frac=0.0):
        e = rng.integers(elo, ehi + 1, size=d).astype(np.float64)
        x = np.where(rng.random(d) < 0.5, -1.0, 1.0) * (1.0 + rng.random(d)) * np.exp2(e)
        x[rng.random(d) < zero_frac] = 0.0
        return x

    rows = [row(lo, lo + 3) for _ in range(8)] + [row(52, 55) for _ in range(8)]
    rows += [row(lo, 55, 0.1) for _ in range(16)]
    x = torch.tensor(np.array(rows), dtype=torch.float32)
    x = (x.to(torch.bfloat16) if dt == "bf16" else x).cuda()
    xa = np.abs(parity.to_f64(x))
    assert xa.max() <= 2.0**56 and xa[xa > 0].min() >= 2.0**lo
    check_roundtrip(tac_gpu, orc, x, d, 64, b, mode, label=f"range {dt} b={b} m={mode}")


@pytest.mark.parametrize("n", [2, 4, 8, 16, 64, 256])
def test_pairs_next_to_bin_edges(tac_gpu, orc, n):
    """Pairs a small angle (1e-6 .. 1e-2 rad, either side) from a bin edge of
    Alg. 1, theta = (k + 1/2) 2 pi / n: a candidate edge one bin off would be
    decided wrong there, by the fast test or the exact path.  fp32 rows
    x = D H y; the oracle sees the same rounded inputs, every code must match."""
    torch = _torch()
    d, rows = 128, 64
    P = d // 2
    rng = np.random.default_rng(100 + n)
    k = rng.integers(0, n, size=(rows, P))
    delta = rng.choice([1e-6, 1e-5, 1e-4, 1e-3, 1e-2], size=(rows, P)) * rng.choice([-1.0, 1.0], size=(rows, P))
    theta = (k + 0.5) * 2.0 * np.pi / n + delta
    r = 0.5 + rng.random((rows, P))
    y = np.zeros((rows, d))
    y[:, 0::2], y[:, 1::2] = r * np.cos(theta), r * np.sin(theta)
    s = orc.signs(0, 0, 0, d)
    x = (orc.transform(y, np.ones(d, dtype=np.int8)) * s).astype(np.float32)
    st = check_roundtrip(tac_gpu, orc, torch.tensor(x).cuda(), d, n, 8, 0, label=f"near edges n={n}",
                         decode_dtypes=("fp32",))
    assert st["angle_mismatch"] == 0, st


@pytest.mark.parametrize("d,n,b,mode", [(128, 64, 8, 0), (128, 256, 4, 1), (64, 128, 8, 0)])
def test_many_tiles_per_cta_every_row(tac_gpu, orc, d, n, b, mode):
    """Enough rows that every CTA of the persistent grid loops over many tiles
    (exercising the multi-stage cp.async pipeline); every row is compared."""
    import os
    torch = _torch()
    w = workloads.CONFIGS["mistral7b" if d == 128 else "llama1b"]
    rows = 160_000 if d == 128 else 120_000
    x = _rows(w, rows, seed=d + n, layer=3, kv=mode)
    cfg = tac_gpu.layer_cfg(d, n, b, mode, 0, 3, mode)
    cache = tac_gpu.encode(x, cfg)
    y = tac_gpu.decode(cache, cfg)
    torch.cuda.synchronize()
    x64 = parity.to_f64(x)
    s = orc.signs(0, 3, mode, d)
    threads = os.cpu_count() or 1
    ref = _encode_diag_threads(orc, x64, s, n, b, mode, threads)
    k, c, hdr = parity.gpu_codes(orc, cache, rows)
    parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=f"many tiles d{d} n{n}")
    v = orc.decode_threads(k, c, hdr, s, n, b, mode, threads)
    parity.compare_decode(parity.to_f64(y), v, "bf16", label=f"many tiles decode d{d} n{n}")


def _encode_diag_threads(orc, x64, s, n, b, mode, threads):
    """The oracle's encode with diagnostics, split over host threads by rows."""
    import threading
    parts = np.array_split(np.arange(x64.shape[0]), threads)
    out = [None] * len(parts)

    def work(i, idx):
        out[i] = orc.encode(x64[idx[0]: idx[-1] + 1], s, n, b, mode)

    ts = [threading.Thread(target=work, args=(i, p)) for i, p in enumerate(parts) if len(p)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    return {key: np.concatenate([o[key] for o in out if o is not None]) for key in out[0]}


@pytest.mark.parametrize("dt", ["bf16", "fp32"])
@pytest.mark.parametrize("b,mode", [(8, 0), (4, 1), (32, 2)])
def test_nonfinite_rows(tac_gpu, orc, dt, b, mode):
    """Rows holding a NaN or an infinity: every code 0 and the header (NaN, NaN)
    (fp32 norms: NaN), a NaN row on decode, TAC_E_NONFINITE in the status word;
    the other rows of the call are unaffected, and an all-finite call leaves the
    status word alone."""
    torch = _torch()
    d, n, layer, kv = 128, 64, 1, mode % 2
    w = workloads.CONFIGS["mistral7b"]
    x = _rows(w, 70, seed=11, dtype=torch.float32, layer=layer, kv=kv).clone()
    bad = np.array([3, 17, 40, 69])
    x[3, 5] = float("nan")
    x[17, 100] = float("inf")
    x[40, 0] = float("-inf")
    x[69, :] = float("nan")
    x = (x.to(torch.bfloat16) if dt == "bf16" else x).contiguous()
    good = np.setdiff1d(np.arange(x.shape[0]), bad)
    cfg = tac_gpu.layer_cfg(d, n, b, mode, 0, layer, kv)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    cache = tac_gpu.encode(x, cfg, status=status)
    y = tac_gpu.decode(cache, cfg, dtype=torch.float32)
    torch.cuda.synchronize()
    assert int(status.item()) == tac_gpu.TAC_E_NONFINITE
    k, c, hdr = parity.gpu_codes(orc, cache, x.shape[0])
    assert np.all(k[bad] == 0)
    if mode == parity.FP32_MODE:
        assert np.all(np.isnan(np.ascontiguousarray(c[bad], dtype=np.int32).view(np.float32)))
    else:
        assert np.all(c[bad] == 0) and np.all(np.isnan(hdr[bad]))
    yb = parity.to_f64(y)[bad]
    assert np.all(np.isnan(yb)), yb[:, :4]
    # the finite rows of the same call match the oracle
    x64 = parity.to_f64(x)[good]
    s = orc.signs(0, layer, kv, d)
    ref = orc.encode(x64, s, n, b, mode)
    parity.compare_encode(orc, x64, ref, k[good], c[good], hdr[good] if hdr is not None else None, n, b, mode,
                          label=f"finite rows beside non-finite ones {dt} b={b} m={mode}")
    # an all-finite call leaves the status word as it is
    status.zero_()
    tac_gpu.encode(x[torch.from_numpy(good).cuda()].contiguous(), cfg, status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0


@pytest.mark.parametrize("room", ["min", "partial"])
def test_small_workspace_rows_redecided_whole(tac_gpu, orc, room):
    """With the minimum workspace (no queue room) every queued code's row is
    re-decided whole through the bitmap; with a queue of a few dozen entries
    some codes go through the queue and the rest of the rows whole.  The
    records satisfy the same parity rule as with the recommended workspace."""
    torch = _torch()
    w = workloads.CONFIGS["mistral7b"]
    for kv in (workloads.K, workloads.V):
        d, n, b, mode = w.codebook(0, kv)
        x = _rows(w, 6000, seed=5, layer=0, kv=kv)
        cfg = tac_gpu.layer_cfg(d, n, b, mode, 0, 0, kv)
        cache = tac_gpu.Cache.empty(cfg, x.shape[0])
        jobs = [tac_gpu.EncodeJob(cfg, x, cache)]
        rec, mn = tac_gpu.encode_workspace_bytes(jobs)
        size = mn if room == "min" else mn + 32 * 40
        wsb = torch.empty(size, dtype=torch.uint8, device="cuda")
        tac_gpu.encode_multi(jobs, workspace=wsb)
        torch.cuda.synchronize()
        x64 = parity.to_f64(x)
        s = orc.signs(0, 0, kv, d)
        ref = orc.encode(x64, s, n, b, mode)
        k, c, hdr = parity.gpu_codes(orc, cache, x.shape[0])
        parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=f"workspace {room} kv={kv}")
        # the queue overflowed: the counter passed the queue's capacity
        appended = int(wsb[:8].cpu().numpy().view(np.uint64)[0])
        assert appended > (0 if room == "min" else 40), appended
