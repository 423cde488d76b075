"""tac_attend_multi_static: attention with the library's static device
workspace, for callers that cannot allocate.

The file is named to be collected last, so that on a full run the static
array has already served the earlier attention tests' kernels (it must not
depend on what the array held before), and it passes on its own too.

GPU check: two different job sets in a row through the static entry point give
the same bits as tac_attend_multi with a fresh caller workspace (same kernels,
same grouping, same partial-record layout), and the first set run again after
the second still does (nothing carried over in the array).
CPU checks: argument checks and the size limit happen before any device work.
"""
import math
import os
import re

import pytest

import workloads

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _host_job(tac, d=128, nq=4, tokens=1000, capacity=None):
    j = tac._AttJob()
    j.cfg_k = tac.LayerCfg(d, 64, 8, 0).to_c()
    j.cfg_v = tac.LayerCfg(d, 64, 4, 1).to_c()
    j.k_codes = j.k_norms = j.v_codes = j.v_norms = 4096
    j.capacity, j.tokens = capacity or tokens, tokens
    j.q.data, j.q.dtype, j.q.rows, j.q.row_stride = 8192, 0, nq, d
    j.out.data, j.out.dtype, j.out.rows, j.out.row_stride = 16384, 0, nq, d
    j.scale = 0.088
    return j


def test_static_workspace_size_matches_header(tac_host):
    """The binding's limit is the header's TAC_ATTEND_STATIC_WS_BYTES."""
    src = open(os.path.join(ROOT, "include", "tac.h")).read()
    m = re.search(r"#define\s+TAC_ATTEND_STATIC_WS_BYTES\s+\((\d+)\s*<<\s*(\d+)\)", src)
    assert m, "TAC_ATTEND_STATIC_WS_BYTES not found"
    assert int(m.group(1)) << int(m.group(2)) == tac_host.ATTEND_STATIC_WS_BYTES


def test_static_rejects_oversize_and_bad_jobs(tac_host):
    """Jobs needing more than the static array are refused with
    TAC_E_UNSUPPORTED and a message naming both sizes; bad jobs with
    TAC_E_INVAL, as in tac_attend_multi; nothing reaches the device."""
    lib = tac_host.load()
    limit = tac_host.ATTEND_STATIC_WS_BYTES
    # ceil(T / 256) * 8 * 130 floats: the largest T that still fits, and one split more
    per_split = 8 * 130 * 4
    fit_splits = limit // per_split
    big = (tac_host._AttJob * 1)(_host_job(tac_host, nq=8, tokens=(fit_splits + 1) * 256))
    need = lib.tac_attend_workspace_bytes(big, 1)
    assert need > limit
    assert lib.tac_attend_multi_static(big, 1, None) == tac_host.TAC_E_UNSUPPORTED
    msg = tac_host.last_error()
    assert str(need) in msg and str(limit) in msg, msg
    ok = (tac_host._AttJob * 1)(_host_job(tac_host, nq=8, tokens=fit_splits * 256))
    assert lib.tac_attend_workspace_bytes(ok, 1) <= limit
    # two jobs that fit alone but not together
    two = (tac_host._AttJob * 2)(_host_job(tac_host, nq=8, tokens=fit_splits * 256),
                                 _host_job(tac_host, nq=8, tokens=256))
    assert lib.tac_attend_multi_static(two, 2, None) == tac_host.TAC_E_UNSUPPORTED
    for kw in (dict(nq=0), dict(nq=9), dict(tokens=0), dict(d=32)):
        a = (tac_host._AttJob * 1)(_host_job(tac_host, **kw))
        assert lib.tac_attend_multi_static(a, 1, None) in (tac_host.TAC_E_INVAL, tac_host.TAC_E_UNSUPPORTED), kw
    assert lib.tac_attend_multi_static(None, -1, None) == tac_host.TAC_E_INVAL
    assert lib.tac_attend_multi_static(None, 1, None) == tac_host.TAC_E_INVAL


def _jobs(tac, specs):
    import torch
    jobs = []
    for sp in specs:
        d, T, nq, seed = sp["d"], sp["T"], sp["nq"], sp["seed"]
        tdt = torch.bfloat16 if sp.get("bf16") else torch.float32
        w = workloads.CONFIGS["mistral7b" if d == 128 else "llama1b"]
        heads_T = -(-T // w.heads)
        caches = []
        for kv, (n, b, mode) in ((0, sp["k"]), (1, sp["v"])):
            x = workloads.block(w, 3, kv, tokens=heads_T, seed=seed, device="cuda")[:T].contiguous()
            cfg = tac.layer_cfg(d, n, b, mode, 0, 3, kv)
            caches.append((cfg, tac.encode(x, cfg)))
        g = torch.Generator(device="cuda")
        g.manual_seed(seed)
        q = (torch.randn((nq, d), generator=g, device="cuda") * 0.5).to(tdt)
        out = torch.full((nq, d), float("nan"), dtype=tdt, device="cuda")
        jobs.append(tac.AttendJob(caches[0][0], caches[0][1], caches[1][0], caches[1][1], T, q, out,
                                  1.0 / math.sqrt(d)))
    return jobs


def _outs(jobs):
    return [j.out.clone() for j in jobs]


def _reset(jobs):
    for j in jobs:
        j.out.fill_(float("nan"))


@pytest.mark.gpu
def test_static_matches_workspace_entry_two_calls_in_a_row(tac_gpu):
    import torch
    tac = tac_gpu
    tac.attend_multi_static([])          # first-call setup on this device
    set_a = _jobs(tac, [
        dict(d=128, T=1000, nq=4, k=(64, 8, 0), v=(64, 4, 1), seed=11),
        dict(d=64, T=700, nq=8, k=(256, 32, 2), v=(56, 8, 0), seed=12),
        dict(d=128, T=37, nq=1, k=(48, 4, 1), v=(16, 4, 1), seed=13, bf16=True),
    ])
    set_b = _jobs(tac, [
        dict(d=128, T=3000, nq=8, k=(128, 8, 0), v=(64, 4, 1), seed=21),
        dict(d=64, T=1, nq=2, k=(64, 8, 0), v=(64, 4, 1), seed=22),
    ])
    stream = torch.cuda.current_stream()
    want = {}
    for name, jobs in (("a", set_a), ("b", set_b)):
        ws = torch.empty(tac.attend_workspace_bytes(jobs), dtype=torch.uint8, device="cuda")
        tac.attend_multi(jobs, ws, stream=stream)
        torch.cuda.synchronize()
        want[name] = _outs(jobs)
        assert all(torch.isfinite(o.float()).all() for o in want[name])
        _reset(jobs)
    assert tac.attend_workspace_bytes(set_a + set_b) <= tac.ATTEND_STATIC_WS_BYTES
    for name, jobs in (("a", set_a), ("b", set_b), ("a", set_a)):
        tac.attend_multi_static(jobs, stream=stream)
        torch.cuda.synchronize()
        for got, ref in zip(_outs(jobs), want[name]):
            assert torch.equal(got, ref), name
        _reset(jobs)
