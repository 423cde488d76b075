"""Full-size workloads in the launch configuration the bench times (one batched
launch over every (layer, K/V) block), checked on sampled rows against the oracle
and on properties that hold at any size."""
import math
import os

import numpy as np
import pytest

import parity
import workloads

pytestmark = pytest.mark.gpu


def _torch():
    import torch
    return torch


def _build(tac, w, seed=0):
    torch = _torch()
    xs, caches, cfgs, enc_jobs = {}, {}, {}, []
    for (l, kv) in w.blocks():
        d, n, b, mode = w.codebook(l, kv)
        cfg = tac.layer_cfg(d, n, b, mode, seed, l, kv)
        x = workloads.block(w, l, kv, seed=seed, device="cuda")
        cache = tac.Cache.empty(cfg, x.shape[0])
        xs[(l, kv)], caches[(l, kv)], cfgs[(l, kv)] = x, cache, cfg
        enc_jobs.append(tac.EncodeJob(cfg, x, cache))
    return xs, caches, cfgs, enc_jobs


def _sample(rows, k, rng):
    idx = np.unique(np.concatenate([rng.choice(rows, size=k, replace=False), [0, rows - 1]]))
    return idx


@pytest.mark.parametrize("name", ["llama1b", "mistral7b"])
def test_full_cache_encode_decode_sampled(tac_gpu, orc, name):
    torch = _torch()
    tac = tac_gpu
    w = workloads.CONFIGS[name]
    xs, caches, cfgs, enc_jobs = _build(tac, w)
    tac.encode_multi(enc_jobs)
    ys = {key: torch.empty_like(xs[key]) for key in xs}
    tac.decode_multi([tac.DecodeJob(cfgs[key], caches[key], ys[key]) for key in xs])
    torch.cuda.synchronize()
    rng = np.random.default_rng(1)
    # at least 10^6 codes per workload: 64 blocks x 256 rows x 64 pairs, 32 x 1000 x 32
    per_block = 256 if name == "mistral7b" else 1000
    threads = os.cpu_count() or 1
    tot = {"codes": 0, "angle_mismatch": 0, "norm_mismatch": 0}
    for key in xs:
        d, n, b, mode = w.codebook(*key)
        rows = xs[key].shape[0]
        idx = _sample(rows, per_block, rng)
        it = torch.from_numpy(idx).cuda()
        x64 = parity.to_f64(xs[key][it])
        s = orc.signs(0, key[0], key[1], d)
        ref = orc.encode_threads(x64, s, n, b, mode, threads, diagnostics=True)
        k, c, hdr = parity.gpu_codes(orc, caches[key], slots=idx)
        st = parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=f"{name} {key}")
        for f in tot:
            tot[f] += st[f]
        v = orc.decode_threads(k, c, hdr, s, n, b, mode, threads)
        parity.compare_decode(parity.to_f64(ys[key][it]), v, "bf16", label=f"{name} {key} decode")
    assert tot["codes"] >= 1_000_000
    assert tot["angle_mismatch"] <= 1e-6 * tot["codes"] and tot["norm_mismatch"] <= 1e-6 * tot["codes"], tot


def test_full_cache_properties(tac_gpu):
    """Any size: headers finite with r_min <= r_max; decoded rows finite and, block by
    block, within the quantizer's own error scale of the input."""
    torch = _torch()
    tac = tac_gpu
    w = workloads.CONFIGS["mistral7b"]
    xs, caches, cfgs, enc_jobs = _build(tac, w, seed=2)
    tac.encode_multi(enc_jobs)
    for key in xs:
        cfg = cfgs[key]
        off = tac.header_offset(cfg, caches[key].capacity)
        hdr = caches[key].norms[off: off + 8 * caches[key].capacity].view(torch.float32).view(-1, 2)
        assert bool(torch.isfinite(hdr).all())
        assert bool((hdr[:, 0] <= hdr[:, 1]).all())
        assert bool((hdr[:, 0] >= 0).all())
        y = tac.decode(caches[key], cfg, dtype=torch.float32)
        x = xs[key].float()
        assert bool(torch.isfinite(y).all())
        rel = ((y - x).norm(dim=1) / x.norm(dim=1).clamp_min(1e-30))
        # n >= 64 angles + 8-bit (K) or 4-bit log (V) norms: relative error well below 1
        assert float(rel.mean()) < (0.12 if key[1] == 0 else 0.35), (key, float(rel.mean()))
        del y


def test_append_step_full(tac_gpu, orc):
    """Config 4: 256 sequences x 32 layers x 2 x 8 heads, one token each, encoded in
    one launch into scattered slots of paged per-(layer, kv) pools."""
    torch = _torch()
    tac = tac_gpu
    a = workloads.APPEND
    w = workloads.CONFIGS[a["base"]]
    cap = workloads.append_capacity()
    slots = torch.from_numpy(workloads.append_slots(0, 0)).cuda()
    rows = a["seqs"] * w.heads
    jobs, xs = [], {}
    for (l, kv) in w.blocks():
        d, n, b, mode = w.codebook(l, kv)
        cfg = tac.layer_cfg(d, n, b, mode, 0, l, kv)
        x = workloads.block(w, l, kv, tokens=a["seqs"], seed=11, device="cuda")  # rows = h*T+t
        x = x.view(w.heads, a["seqs"], d).transpose(0, 1).reshape(rows, d).contiguous()  # row = s*H + h
        pool = tac.Cache.empty(cfg, cap)
        jobs.append(tac.EncodeJob(cfg, x, pool, slots))
        xs[(l, kv)] = x
    tac.encode_multi(jobs)
    torch.cuda.synchronize()
    sl = slots.cpu().numpy()
    threads = os.cpu_count() or 1
    for j, key in zip(jobs, list(xs)):   # every block: 64 x 2048 rows, 8.4e6 codes
        d, n, b, mode = w.codebook(*key)
        x64 = parity.to_f64(j.x)
        ref = orc.encode_threads(x64, orc.signs(0, key[0], key[1], d), n, b, mode, threads, diagnostics=True)
        k, c, hdr = parity.gpu_codes(orc, j.cache, slots=sl)
        parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=f"append {key}")


def test_longctx_decode_sweep_sampled(tac_gpu, orc):
    """Config 5 shape (4 heads x 131072 tokens per (layer, kv)) on layers 0, 13,
    27: every n of the sweep for K and for V (K and V are coded independently,
    so this covers all 25 (n_K, n_V) pairs), each whole block encoded and
    decoded, 400 rows of each compared with the oracle."""
    torch = _torch()
    tac = tac_gpu
    w = workloads.CONFIGS["longctx"]
    rng = np.random.default_rng(3)
    threads = os.cpu_count() or 1
    for layer in (0, 13, 27):
        for kv in (0, 1):
            x = workloads.block(w, layer, kv, seed=5, device="cuda")
            b, mode = (8, 0) if kv == 0 else (4, 1)
            s = orc.signs(0, layer, kv, 128)
            for n in workloads.SWEEP_N:
                cfg = tac.layer_cfg(128, n, b, mode, 0, layer, kv)
                cache = tac.encode(x, cfg)
                y = tac.decode(cache, cfg)
                torch.cuda.synchronize()
                idx = _sample(x.shape[0], 400, rng)
                it = torch.from_numpy(idx).cuda()
                k, c, hdr = parity.gpu_codes(orc, cache, slots=idx)
                v = orc.decode(k, c, hdr, s, n, b, mode)
                parity.compare_decode(parity.to_f64(y[it]), v, "bf16", label=f"longctx L{layer} kv{kv} n={n}")
                x64 = parity.to_f64(x[it])
                ref = orc.encode_threads(x64, s, n, b, mode, threads, diagnostics=True)
                parity.compare_encode(orc, x64, ref, k, c, hdr, n, b, mode, label=f"longctx enc L{layer} kv{kv} n={n}")
                del y, cache
            del x


def test_full_cache_attention_sampled(tac_gpu, orc):
    """Attention from the records at the bench's size and launch configuration
    (`bench.py --config attend`: 32 layers x 8 KV heads x 32768 tokens, one job
    per (layer, head), 4 query rows, one tac_attend_multi call): every output
    finite, sampled jobs equal to fp64 softmax attention over the oracle's
    decode of their records within the bound of tests/test_gpu_attend.py."""
    torch = _torch()
    tac = tac_gpu
    w = workloads.CONFIGS["mistral7b"]
    T, nq = w.tokens, 4
    caches, jobs = {}, []
    for l in range(w.layers):
        for kv in (workloads.K, workloads.V):
            d, n, b, mode = w.codebook(l, kv)
            cfg = tac.layer_cfg(d, n, b, mode, 0, l, kv)
            x = workloads.block(w, l, kv, device="cuda", dtype=torch.bfloat16)
            for h in range(w.heads):
                caches[(l, kv, h)] = (cfg, tac.encode(x[h * T:(h + 1) * T], cfg))
            del x
        for h in range(w.heads):
            g = torch.Generator(device="cuda")
            g.manual_seed(l * 64 + h)
            q = torch.randn((nq, w.d), generator=g, device="cuda").to(torch.bfloat16)
            (kc, kk), (vc, vk) = caches[(l, workloads.K, h)], caches[(l, workloads.V, h)]
            jobs.append(((l, h), tac.AttendJob(kc, kk, vc, vk, T, q, torch.empty_like(q), 1.0 / math.sqrt(w.d))))
    tac.attend_multi([j for _, j in jobs])
    torch.cuda.synchronize()
    for _, j in jobs:
        assert torch.isfinite(j.out.float()).all()
    picks = {(0, 0), (17, 3), (31, 7)}
    for (l, h), j in jobs:
        if (l, h) not in picks:
            continue
        dec = []
        for kv in (workloads.K, workloads.V):
            cfg, cache = caches[(l, kv, h)]
            k, c, hdr = parity.gpu_codes(orc, cache, T)
            if hdr is None:
                hdr = np.zeros((T, 2), dtype=np.float32)
            dec.append(orc.decode(k, c, hdr, parity.signs_pm1(cfg.signs, cfg.d), cfg.n_angle, cfg.norm_bits,
                                  cfg.norm_mode))
        kh, vh = dec
        q64 = parity.to_f64(j.q)
        want = orc.attend(q64, kh, vh, j.scale)
        tol = (2.0**-11 * j.scale * np.linalg.norm(q64, axis=1, keepdims=True) * np.linalg.norm(kh, axis=1).max()
               + 2.0**-16) * np.abs(vh).max() + parity.bf16_half_ulp(want)
        err = np.abs(parity.to_f64(j.out) - want)
        assert np.all(err <= tol), ((l, h), float((err / tol).max()))
