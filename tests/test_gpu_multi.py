"""Batched launches (tac_encode_multi / tac_decode_multi): mixed codebooks, d and
dtypes in one call, scatter-append into record slots, gather decode."""
import numpy as np
import pytest

import parity
import workloads

pytestmark = pytest.mark.gpu


def _torch():
    import torch
    return torch


def _same_planes(a, b):
    """Records equal plane by plane (bytes between the norm and header planes are padding)."""
    for pa, pb in zip(a.planes(), b.planes()):
        assert np.array_equal(pa.view(np.uint8), pb.view(np.uint8))


def _jobs_spec():
    # (d, n, b, mode, dtype, rows, layer, kv)
    return [(128, 256, 8, 0, "bf16", 700, 0, 0), (128, 64, 4, 1, "bf16", 300, 0, 1),
            (128, 16, 8, 1, "bf16", 129, 5, 0), (64, 128, 8, 0, "bf16", 513, 1, 0),
            (64, 64, 4, 1, "fp32", 257, 1, 1), (128, 2, 4, 0, "fp32", 64, 9, 1),
            (32, 8, 8, 0, "bf16", 100, 2, 0), (16, 32, 4, 1, "fp32", 90, 3, 1)]


def _make_x(d, dtype, rows, seed):
    torch = _torch()
    w = workloads.CONFIGS["mistral7b"]
    x = workloads.block(w, seed % 32, seed % 2, tokens=-(-rows // w.heads), seed=seed, device="cuda")[:rows, :d]
    return x.to(torch.bfloat16 if dtype == "bf16" else torch.float32).contiguous()


def test_encode_multi_equals_single_calls(tac_gpu, orc):
    torch = _torch()
    tac = tac_gpu
    jobs, singles = [], []
    for i, (d, n, b, mode, dt, rows, layer, kv) in enumerate(_jobs_spec()):
        cfg = tac.layer_cfg(d, n, b, mode, 0, layer, kv)
        x = _make_x(d, dt, rows, i)
        jobs.append(tac.EncodeJob(cfg, x, tac.Cache.empty(cfg, rows)))
        singles.append(tac.encode(x, cfg))
    for j in jobs:
        j.cache.codes.zero_(); j.cache.norms.zero_()
    tac.encode_multi(jobs)
    torch.cuda.synchronize()
    for j, s in zip(jobs, singles):
        _same_planes(j.cache, s)
    # and the batched output is oracle-exact too (codes and headers)
    j = jobs[0]
    x64 = parity.to_f64(j.x)
    ref = orc.encode(x64, orc.signs(0, 0, 0, 128), 256, 8, 0)
    k, c, hdr = parity.gpu_codes(orc, j.cache, 700)
    parity.compare_encode(orc, x64, ref, k, c, hdr, 256, 8, 0, label="multi job0")


def test_decode_multi_equals_single_calls(tac_gpu):
    torch = _torch()
    tac = tac_gpu
    jobs, singles = [], []
    for i, (d, n, b, mode, dt, rows, layer, kv) in enumerate(_jobs_spec()):
        cfg = tac.layer_cfg(d, n, b, mode, 0, layer, kv)
        cache = tac.encode(_make_x(d, dt, rows, i), cfg)
        out_dt = torch.float32 if i % 2 else torch.bfloat16
        y = torch.full((rows, d), float("nan"), dtype=out_dt, device="cuda")
        jobs.append(tac.DecodeJob(cfg, cache, y))
        singles.append(tac.decode(cache, cfg, dtype=out_dt))
    tac.decode_multi(jobs)
    torch.cuda.synchronize()
    for j, s in zip(jobs, singles):
        assert torch.equal(j.y, s)


def test_scatter_append_and_gather(tac_gpu, orc):
    """Config-4 style step: rows go to scattered record slots of a larger pool;
    untouched slots keep their bytes; a gather decode reads them back."""
    torch = _torch()
    tac = tac_gpu
    rng = np.random.default_rng(0)
    cap, rows = 4096, 1000
    for (n, b, mode) in ((256, 8, 0), (64, 4, 1), (32, 8, 1)):
        cfg = tac.layer_cfg(128, n, b, mode, 0, 3, mode)
        x = _make_x(128, "bf16", rows, n)
        slots = rng.choice(cap, size=rows, replace=False).astype(np.int64)
        pool = tac.Cache.empty(cfg, cap)
        pool.codes.fill_(0xAB); pool.norms.fill_(0xCD)
        before_c, before_n = pool.codes.clone(), pool.norms.clone()
        st = torch.from_numpy(slots).cuda()
        tac.encode_multi([tac.EncodeJob(cfg, x, pool, st)])
        ref = tac.encode(x, cfg)
        torch.cuda.synchronize()
        rc, rn, rh = ref.planes()
        pc, pn, ph = pool.planes()
        assert np.array_equal(pc[slots], rc) and np.array_equal(pn[slots], rn) and np.array_equal(ph[slots], rh)
        untouched = np.setdiff1d(np.arange(cap), slots)
        bc, bn, bh = tac.Cache(cfg, cap, before_c, before_n).planes()
        assert np.array_equal(pc[untouched], bc[untouched]) and np.array_equal(pn[untouched], bn[untouched])
        assert np.array_equal(ph[untouched].view(np.uint32), bh[untouched].view(np.uint32))
        # gather decode of the pool at the same slots == plain decode of the dense records
        y = torch.empty((rows, 128), dtype=torch.bfloat16, device="cuda")
        tac.decode_multi([tac.DecodeJob(cfg, pool, y, st)])
        y_ref = tac.decode(ref, cfg)
        torch.cuda.synchronize()
        assert torch.equal(y, y_ref)


def test_out_of_range_slots_are_skipped(tac_gpu):
    torch = _torch()
    tac = tac_gpu
    cfg = tac.layer_cfg(128, 64, 8, 0)
    x = _make_x(128, "bf16", 4, 1)
    pool = tac.Cache.empty(cfg, 8)
    pool.codes.fill_(7); pool.norms.fill_(9)
    st = torch.tensor([0, -1, 8, 1 << 40], dtype=torch.int64, device="cuda")
    tac.encode_multi([tac.EncodeJob(cfg, x, pool, st)])
    torch.cuda.synchronize()
    c, n, h = pool.planes()
    assert np.all(c[1:] == 7) and np.all(n[1:] == 9)
    assert not np.all(c[0] == 7)
    y = torch.full((4, 128), 5.0, dtype=torch.float32, device="cuda")
    tac.decode_multi([tac.DecodeJob(cfg, pool, y, st)])
    torch.cuda.synchronize()
    assert torch.all(y[1:] == 0)


def test_many_jobs_split_across_launches(tac_gpu):
    """More jobs than one launch holds (TAC_MAX_JOBS) are split transparently."""
    torch = _torch()
    tac = tac_gpu
    jobs, refs = [], []
    for i in range(150):
        cfg = tac.layer_cfg(64, 2 ** (1 + i % 8), 8 if i % 2 else 4, i % 2, 0, i // 2, i % 2)
        x = _make_x(64, "bf16", 1 + (i * 37) % 200, i)
        jobs.append(tac.EncodeJob(cfg, x, tac.Cache.empty(cfg, x.shape[0])))
        refs.append(tac.encode(x, cfg))
    tac.encode_multi(jobs)
    torch.cuda.synchronize()
    for j, r in zip(jobs, refs):
        _same_planes(j.cache, r)
