"""Host-side checks of libtac's C ABI (no GPU needed): the library loads, exports
every entry point include/tac.h declares, validates arguments before touching
the device, and its host functions (signs, plane geometry, rates) agree with the
oracle's independent implementations and the paper's printed rates."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _declared_symbols():
    src = open(os.path.join(ROOT, "include", "tac.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(tac_[a-z0-9_]+)\s*\(", src)))


def test_header_declares_the_path(tac_host):
    syms = _declared_symbols()
    for name in ("tac_make_signs", "tac_encode", "tac_decode", "tac_encode_multi", "tac_decode_multi",
                 "tac_fwht_debug", "tac_last_error"):
        assert name in syms


def test_library_exports_every_declared_symbol(tac_host):
    lib = ctypes.CDLL(tac_host.library_path())
    missing = [s for s in _declared_symbols() if not hasattr(lib, s)]
    assert not missing, missing


def test_version(tac_host):
    assert "libtac" in tac_host.version()


@pytest.mark.parametrize("seed,layer,kv,d,shared", [(0, 0, 0, 128, False), (0, 31, 1, 128, False),
                                                    (12345, 7, 0, 64, False), (2**63 + 5, 3, 1, 16, False),
                                                    (9, 4, 1, 128, True)])
def test_signs_match_oracle(tac_host, orc, seed, layer, kv, d, shared):
    words = tac_host.make_signs(seed, layer, kv, d, shared)
    bits = np.array([(int(words[j // 32]) >> (j % 32)) & 1 for j in range(d)])
    want = orc.signs(seed, layer, kv, d, shared=shared)
    assert np.array_equal(np.where(bits == 1, -1, 1).astype(np.int8), want)


def test_plane_geometry(tac_host):
    for d in (16, 32, 64, 128):
        for n in (2, 4, 16, 64, 128, 256):
            for b, mode in ((8, 0), (4, 1)):
                cfg = tac_host.LayerCfg(d, n, b, mode)
                w = int(math.log2(n))
                assert tac_host.angle_row_bytes(cfg) == d // 2 * w // 8
                assert tac_host.norm_row_bytes(cfg) == d // 2 * b // 8
                for cap in (0, 1, 7, 128, 1000):
                    off = tac_host.header_offset(cfg, cap)
                    assert off % 16 == 0 and off >= cap * (d // 2 * b // 8) and off - cap * d // 2 * b // 8 < 16
                    assert tac_host.norms_bytes(cfg, cap) == off + 8 * cap
                    assert tac_host.codes_bytes(cfg, cap) == cap * (d // 2 * w // 8)


def test_plane_geometry_extra_shapes(tac_host):
    """n = 48, 56 (Table 1) store ceil(log2 n) = 6 bits per code; fp32 norms
    (Sec. 3.1) store 4 bytes per pair and no header plane."""
    for d in (16, 32, 64, 128):
        for n in (48, 56):
            cfg = tac_host.LayerCfg(d, n, 8, 0)
            assert tac_host.angle_row_bytes(cfg) == d // 2 * 6 // 8
        for n in (16, 56, 256):
            cfg = tac_host.LayerCfg(d, n, 32, tac_host.NORM_FP32)
            assert tac_host.norm_row_bytes(cfg) == d // 2 * 4
            for cap in (0, 1, 7, 1000):
                off = tac_host.header_offset(cfg, cap)
                assert off == (cap * d // 2 * 4 + 15) // 16 * 16
                assert tac_host.norms_bytes(cfg, cap) == off
    r = tac_host.rates(128, [56] * 4, [48] * 4, 32, 32)
    assert abs(r["angle_bits"] - (math.log2(56) + math.log2(48)) / 4) < 1e-12
    assert abs(r["total_bits"] - (r["angle_bits"] + 16)) < 1e-12 and r["stored_angle_bits"] == 3.0


def test_record_bytes_match_rate_accounting(tac_host, orc):
    # Eq. 3 total bits per element x d / 8 = record bytes per row (angle + norm + 8-byte header)
    for n in (16, 64, 256):
        for b in (4, 8):
            cfg = tac_host.LayerCfg(128, n, b, 0)
            rec = tac_host.angle_row_bytes(cfg) + tac_host.norm_row_bytes(cfg) + 8
            assert rec * 8 / 128 == orc.total_bits(math.log2(n) / 2, b, 128)


def test_rates_agree_with_oracle(tac_host, orc):
    rng = np.random.default_rng(0)
    for _ in range(20):
        L = int(rng.integers(1, 48))
        nk = [int(2 ** rng.integers(1, 9)) for _ in range(L)]
        nv = [int(2 ** rng.integers(1, 9)) for _ in range(L)]
        assert abs(tac_host.avg_angle_bits(nk, nv) - orc.avg_angle_bits(nk, nv)) < 1e-12
    assert tac_host.total_bits(3.25, 6, 128) == 6.75


def test_early_boost_schedule(tac_host):
    nk, nv = tac_host.early_boost(32, 4, (256, 128), (128, 64))
    assert abs(tac_host.avg_angle_bits(nk, nv) - 3.3125) < 1e-12
    r = tac_host.rates(128, *tac_host.early_boost(32, 4, (256, 256), (64, 64)))
    # Mistral-7B-shaped config: (4 * 4 + 28 * 3) / 32 = 3.125 angle bits; + 3 norm + 0.5 header
    assert abs(r["angle_bits"] - 3.125) < 1e-12 and abs(r["total_bits"] - 6.625) < 1e-12


def _cfg(tac, d=128, n=64, b=8, mode=0):
    return tac.LayerCfg(d, n, b, mode).to_c()


def test_invalid_arguments_rejected_before_launch(tac_host):
    lib = tac_host.load()
    rows = tac_host._Rows()
    rows.data, rows.dtype, rows.rows, rows.row_stride = 16, 0, 4, 128
    buf = 4096
    cases = [
        (dict(d=100), tac_host.TAC_E_INVAL),
        (dict(d=256), tac_host.TAC_E_UNSUPPORTED),
        (dict(n=3), tac_host.TAC_E_UNSUPPORTED),
        (dict(n=24), tac_host.TAC_E_UNSUPPORTED),
        (dict(n=0), tac_host.TAC_E_INVAL),
        (dict(n=512), tac_host.TAC_E_UNSUPPORTED),
        (dict(b=5), tac_host.TAC_E_UNSUPPORTED),
        (dict(b=0), tac_host.TAC_E_INVAL),
        (dict(b=32), tac_host.TAC_E_INVAL),
        (dict(mode=2, b=8), tac_host.TAC_E_INVAL),
        (dict(mode=7), tac_host.TAC_E_INVAL),
    ]
    for kw, want in cases:
        c = _cfg(tac_host, **kw)
        assert lib.tac_encode(ctypes.byref(rows), ctypes.byref(c), buf, buf, None) == want, kw
        assert tac_host.last_error()
    c = _cfg(tac_host)
    bad = tac_host._Rows()
    for field, val in (("dtype", 9), ("rows", -1), ("row_stride", 64), ("data", 8), ("data", 0)):
        bad.data, bad.dtype, bad.rows, bad.row_stride = 16, 0, 4, 128
        setattr(bad, field, val)
        assert lib.tac_encode(ctypes.byref(bad), ctypes.byref(c), buf, buf, None) == tac_host.TAC_E_INVAL, field
    # stride * sizeof(bf16) not a multiple of 16
    bad.data, bad.dtype, bad.rows, bad.row_stride = 16, 0, 4, 132
    assert lib.tac_encode(ctypes.byref(bad), ctypes.byref(c), buf, buf, None) == tac_host.TAC_E_INVAL
    # misaligned planes
    assert lib.tac_encode(ctypes.byref(rows), ctypes.byref(c), buf + 8, buf, None) == tac_host.TAC_E_INVAL
    assert lib.tac_encode(ctypes.byref(rows), ctypes.byref(c), None, buf, None) == tac_host.TAC_E_INVAL
    # decode side
    assert lib.tac_decode(buf, buf, ctypes.byref(_cfg(tac_host, n=3)), ctypes.byref(rows), None) == tac_host.TAC_E_UNSUPPORTED
    # batched: negative count, NULL jobs, capacity too small without slots
    assert lib.tac_encode_multi(None, -1, None) == tac_host.TAC_E_INVAL
    assert lib.tac_encode_multi(None, 2, None) == tac_host.TAC_E_INVAL
    jobs = (tac_host._EncJob * 1)()
    jobs[0].cfg = c
    jobs[0].x = rows
    jobs[0].codes, jobs[0].norms, jobs[0].capacity, jobs[0].slot = buf, buf, 3, None
    assert lib.tac_encode_multi(jobs, 1, None) == tac_host.TAC_E_INVAL
    jobs[0].capacity, jobs[0].slot = 10, buf + 4  # misaligned slot array
    assert lib.tac_encode_multi(jobs, 1, None) == tac_host.TAC_E_INVAL
    # debug transform
    s = (ctypes.c_uint32 * 4)()
    assert lib.tac_fwht_debug(ctypes.byref(rows), 3, s, buf, None) == tac_host.TAC_E_INVAL
    assert lib.tac_fwht_debug(ctypes.byref(rows), 256, s, buf, None) == tac_host.TAC_E_INVAL
    # signs
    assert lib.tac_make_signs(0, 0, 2, 64, s) == tac_host.TAC_E_INVAL
    assert lib.tac_make_signs(0, -1, 0, 64, s) == tac_host.TAC_E_INVAL
    assert lib.tac_make_signs(0, 0, 0, 0, s) == tac_host.TAC_E_INVAL
    assert lib.tac_make_signs_shared(0, 0, s) == tac_host.TAC_E_INVAL


def test_encode_workspace_size_and_checks(tac_host):
    """tac_encode_workspace_bytes: per launch group a 64-byte counter block,
    one bit per warp-tile row (rounded up to 16 bytes) and a copy of its job
    table (104 bytes a job, rounded up to 16) are the minimum; the recommended
    size adds a queue of one 32-byte entry per 512 angle pairs plus 1024.
    tac_encode_multi_ws rejects a NULL, misaligned or too small workspace
    before any device work."""
    lib = tac_host.load()
    rows = tac_host._Rows()
    rows.data, rows.dtype, rows.rows, rows.row_stride = 16, 0, 1000, 128
    buf = 4096
    jobs = (tac_host._EncJob * 2)()
    for i, (n, b) in enumerate(((64, 8), (256, 4))):   # two kernel shapes: two groups
        jobs[i].cfg = _cfg(tac_host, n=n, b=b, mode=i)
        jobs[i].x = rows
        jobs[i].codes, jobs[i].norms, jobs[i].capacity, jobs[i].slot = buf, buf, 1000, None
    mn = ctypes.c_int64(0)
    rec = lib.tac_encode_workspace_bytes(jobs, 2, ctypes.byref(mn))
    per_min = 64 + ((250 * 4 + 127) // 128) * 16 + 112    # d = 128: 4-row warp tiles; one job
    assert mn.value == 2 * per_min
    assert rec == 2 * (per_min + 32 * (1000 * 64 // 512 + 1024))
    assert lib.tac_encode_workspace_bytes(jobs, 2, None) == rec
    assert lib.tac_encode_workspace_bytes(None, 2, None) == -1
    assert lib.tac_encode_multi_ws(jobs, 2, None, rec, None) == tac_host.TAC_E_INVAL
    assert lib.tac_encode_multi_ws(jobs, 2, buf + 8, rec, None) == tac_host.TAC_E_INVAL
    assert lib.tac_encode_multi_ws(jobs, 2, buf, mn.value - 16, None) == tac_host.TAC_E_INVAL
    assert lib.tac_encode_multi_ws(None, 0, None, 0, None) == tac_host.TAC_OK
    assert lib.tac_encode_workspace_bytes(None, 0, ctypes.byref(mn)) == 0 and mn.value == 0


def test_empty_calls_succeed_without_device(tac_host):
    lib = tac_host.load()
    rows = tac_host._Rows()
    rows.data, rows.dtype, rows.rows, rows.row_stride = 0, 0, 0, 128
    c = _cfg(tac_host)
    assert lib.tac_encode(ctypes.byref(rows), ctypes.byref(c), None, None, None) == tac_host.TAC_OK
    assert lib.tac_decode(None, None, ctypes.byref(c), ctypes.byref(rows), None) == tac_host.TAC_OK
    assert lib.tac_encode_multi(None, 0, None) == tac_host.TAC_OK
    assert lib.tac_decode_multi(None, 0, None) == tac_host.TAC_OK


def test_attend_validation_and_workspace_size(tac_host):
    """tac_attend_*: argument checks happen before any device work; the
    workspace holds ceil(tokens/256) * nq * (d + 2) floats per job, each job's
    part rounded up to 16 bytes."""
    lib = tac_host.load()

    def job(d=128, nq=4, tokens=1000, capacity=1000, kn=64, vn=56, vb=4, vmode=1, qdt=0, odt=0, orows=None):
        j = tac_host._AttJob()
        j.cfg_k = tac_host.LayerCfg(d, kn, 8, 0).to_c()
        j.cfg_v = tac_host.LayerCfg(d, vn, vb, vmode).to_c()
        j.k_codes = j.k_norms = j.v_codes = j.v_norms = 4096
        j.capacity, j.tokens = capacity, tokens
        j.q.data, j.q.dtype, j.q.rows, j.q.row_stride = 8192, qdt, nq, d
        j.out.data, j.out.dtype, j.out.rows, j.out.row_stride = 16384, odt, nq if orows is None else orows, d
        j.scale = 0.088
        return j

    arr = (tac_host._AttJob * 2)(job(), job(d=64, nq=1, tokens=257, capacity=300, vn=256, vb=32, vmode=2))
    want = (math.ceil(1000 / 256) * 4 * 130 + 3) // 4 * 4 * 4 + (2 * 1 * 66 + 3) // 4 * 4 * 4
    assert lib.tac_attend_workspace_bytes(arr, 2) == want
    bad = [dict(nq=0), dict(nq=9), dict(tokens=0), dict(tokens=1001), dict(orows=3), dict(odt=1),
           dict(d=32)]
    for kw in bad:
        a = (tac_host._AttJob * 1)(job(**kw))
        rc = lib.tac_attend_multi(a, 1, 4096, 1 << 30, None)
        assert rc in (tac_host.TAC_E_INVAL, tac_host.TAC_E_UNSUPPORTED), kw
        assert lib.tac_attend_workspace_bytes(a, 1) == -1, kw
    a = (tac_host._AttJob * 1)(job())
    j0 = a[0]
    j0.cfg_v.d = 64
    assert lib.tac_attend_multi(a, 1, 4096, 1 << 30, None) == tac_host.TAC_E_INVAL   # K and V d differ
    a = (tac_host._AttJob * 1)(job())
    assert lib.tac_attend_multi(a, 1, 4096, 16, None) == tac_host.TAC_E_INVAL        # workspace too small
    assert lib.tac_attend_multi(a, 1, 4100, 1 << 30, None) == tac_host.TAC_E_INVAL   # misaligned workspace
    assert lib.tac_attend_multi(None, 0, None, 0, None) == tac_host.TAC_OK


def test_binding_constants_match_header(tac_host):
    """The binding's copies of the header's limits agree with include/tac.h."""
    import os
    import re
    src = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "tac.h")).read()

    def define(name):
        m = re.search(r"#define\s+" + name + r"\s+(\d+)\b", src)
        assert m, name
        return int(m.group(1))

    assert define("TAC_MAX_JOBS") == tac_host.MAX_JOBS
    assert define("TAC_ATTEND_MAX_JOBS") == tac_host.ATTEND_MAX_JOBS
    assert define("TAC_ATTEND_SPLIT") == 256


def test_launch_count_matches_the_grouping(tac_host):
    """launch_count (the bench's gpu_launches): jobs with rows grouped by kernel
    shape (d, dtype, n, norm bits, norm mode), at most MAX_JOBS to a group; an
    encode group launches the encode kernel and its fix-up, a decode group one
    kernel."""
    import torch
    tac = tac_host
    k_cfg, v_cfg = tac.LayerCfg(128, 64, 8, 0), tac.LayerCfg(128, 256, 4, 1)
    x = torch.zeros((4, 128), dtype=torch.bfloat16)
    empty = torch.zeros((0, 128), dtype=torch.bfloat16)
    enc = [tac.EncodeJob(k_cfg, x, None), tac.EncodeJob(k_cfg, x, None), tac.EncodeJob(v_cfg, x, None),
           tac.EncodeJob(v_cfg, empty, None), tac.EncodeJob(k_cfg, x.float(), None)]
    assert tac.launch_count(enc) == 2 * 3            # (k, bf16), (v, bf16), (k, fp32); the empty job adds none
    many = [tac.EncodeJob(k_cfg, x, None)] * (tac.MAX_JOBS + 1)
    assert tac.launch_count(many) == 2 * 2
    dec = [tac.DecodeJob(k_cfg, None, x), tac.DecodeJob(v_cfg, None, x), tac.DecodeJob(v_cfg, None, empty)]
    assert tac.launch_count(dec) == 2
    assert tac.launch_count([]) == 0
