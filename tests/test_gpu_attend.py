"""Attention straight from records (tac_attend_multi) vs the oracle (GB300).

The oracle decodes the GPU's own K and V records (orc.decode, fp64 dense H)
and runs plain softmax attention over them (orc.attend), so the comparison
isolates the rotated-domain attention: scores against H D q, values
accumulated as y^ and transformed back once.

Tolerance (fp32 arithmetic on the GPU): every score is an fp32 sum of 64
products of the rotated query with r^ (cos, sin), the rotated query carries the
butterfly's rounding, the table 1 ulp; all of it is far below
2^-12 * scale * ||q|| * max_t ||k^_t|| (the Cauchy-Schwarz bound on |s_t|
times 2^-12).  A score error e changes the softmax weights by at most ~2e in
total variation, so |out_gpu - out| <= (2^-11 * scale ||q|| max ||k^|| + 2^-16)
* max_t |v^_t|_inf, plus half a bf16 ulp for bf16 outputs.  A wrong bin,
centre, sign, norm or transform gives errors of order max |v^|.
"""
import math

import numpy as np
import pytest

import parity
import workloads

pytestmark = pytest.mark.gpu


def _cache(tac, x, d, n, b, mode, layer, kv):
    cfg = tac.layer_cfg(d, n, b, mode, 0, layer, kv)
    return cfg, tac.encode(x, cfg)


def _oracle_rows(orc, tac, cfg, cache, tokens):
    k, c, hdr = parity.gpu_codes(orc, cache, tokens)
    if hdr is None:
        hdr = np.zeros((tokens, 2), dtype=np.float32)
    s = parity.signs_pm1(cfg.signs, cfg.d)
    return orc.decode(k, c, hdr, s, cfg.n_angle, cfg.norm_bits, cfg.norm_mode)


def _check(orc, tac, jobs_spec, dtype="fp32"):
    import torch
    tdt = torch.float32 if dtype == "fp32" else torch.bfloat16
    jobs, refs = [], []
    for sp in jobs_spec:
        d, T, nq, kc, vc, seed = sp["d"], sp["T"], sp["nq"], sp["k"], sp["v"], sp["seed"]
        w = workloads.CONFIGS["mistral7b" if d == 128 else "llama1b"]
        heads_T = -(-T // w.heads)
        xk = workloads.block(w, 2, 0, tokens=heads_T, seed=seed, device="cuda")[:T].contiguous()
        xv = workloads.block(w, 2, 1, tokens=heads_T, seed=seed, device="cuda")[:T].contiguous()
        kcfg, kcache = _cache(tac, xk, d, *kc, 2, 0)
        vcfg, vcache = _cache(tac, xv, d, *vc, 2, 1)
        g = torch.Generator(device="cuda")
        g.manual_seed(seed)
        q = (torch.randn((nq, d), generator=g, device="cuda") * 0.5).to(tdt)
        out = torch.empty((nq, d), dtype=tdt, device="cuda")
        scale = 1.0 / math.sqrt(d)
        jobs.append(tac.AttendJob(kcfg, kcache, vcfg, vcache, T, q, out, scale))
        refs.append((kcfg, kcache, vcfg, vcache, T, q, scale))
    tac.attend_multi(jobs)
    torch.cuda.synchronize()
    for job, (kcfg, kcache, vcfg, vcache, T, q, scale) in zip(jobs, refs):
        kh = _oracle_rows(orc, tac, kcfg, kcache, T)
        vh = _oracle_rows(orc, tac, vcfg, vcache, T)
        q64 = parity.to_f64(q)
        want = orc.attend(q64, kh, vh, scale)
        got = parity.to_f64(job.out)
        kmax = np.linalg.norm(kh, axis=1).max()
        vmax = np.abs(vh).max()
        tol = (2.0**-11 * scale * np.linalg.norm(q64, axis=1, keepdims=True) * kmax + 2.0**-16) * vmax
        if dtype == "bf16":
            tol = tol + parity.bf16_half_ulp(want)
        err = np.abs(got - want)
        assert np.all(err <= tol), (T, q.shape, float((err / tol).max()))


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
@pytest.mark.parametrize("nq", [1, 4, 8])
@pytest.mark.parametrize("T", [1, 300, 1000])
def test_attend_d128(tac_gpu, orc, dtype, nq, T):
    spec = [dict(d=128, T=T, nq=nq, k=(64, 8, 0), v=(64, 4, 1), seed=T + nq)]
    _check(orc, tac_gpu, spec, dtype)


@pytest.mark.parametrize("nq", [2, 3])
@pytest.mark.parametrize("T", [257, 513])
def test_attend_d64(tac_gpu, orc, nq, T):
    spec = [dict(d=64, T=T, nq=nq, k=(128, 8, 0), v=(64, 4, 1), seed=T * nq)]
    _check(orc, tac_gpu, spec)


def test_attend_codebook_mix_and_many_jobs(tac_gpu, orc):
    """Jobs of different codebooks (fp32 norms, n = 56, 256, log / linear norms),
    d and sizes in one call: grouped launches, per-job workspace parts."""
    spec = [
        dict(d=128, T=700, nq=4, k=(256, 32, 2), v=(56, 8, 0), seed=1),
        dict(d=128, T=64, nq=2, k=(48, 4, 1), v=(256, 32, 2), seed=2),
        dict(d=64, T=900, nq=8, k=(64, 8, 0), v=(16, 4, 1), seed=3),
        dict(d=128, T=2048, nq=4, k=(64, 8, 0), v=(64, 4, 1), seed=4),
        dict(d=64, T=5, nq=1, k=(2, 8, 0), v=(4, 4, 0), seed=5),
    ]
    _check(orc, tac_gpu, spec)


def test_attend_prepared_call_matches_direct(tac_gpu):
    """attend_multi_prepared (job array marshalled once, called twice) gives the
    bits of attend_multi."""
    import torch
    tac = tac_gpu
    w = workloads.CONFIGS["mistral7b"]
    jobs = []
    for seed, T in ((7, 777), (8, 33)):
        xk = workloads.block(w, 1, 0, tokens=T, seed=seed, device="cuda")[:T].contiguous()
        xv = workloads.block(w, 1, 1, tokens=T, seed=seed, device="cuda")[:T].contiguous()
        kcfg, kcache = _cache(tac, xk, 128, 128, 8, 0, 1, 0)
        vcfg, vcache = _cache(tac, xv, 128, 64, 4, 1, 1, 1)
        q = torch.randn((4, 128), device="cuda").to(torch.bfloat16)
        jobs.append(tac.AttendJob(kcfg, kcache, vcfg, vcache, T, q, torch.empty_like(q), 0.088))
    tac.attend_multi(jobs)
    torch.cuda.synchronize()
    want = [j.out.clone() for j in jobs]
    call = tac.attend_multi_prepared(jobs)
    for _ in range(2):
        for j in jobs:
            j.out.zero_()
        call()
        torch.cuda.synchronize()
        for j, ref in zip(jobs, want):
            assert torch.equal(j.out, ref)
