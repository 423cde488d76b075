"""Prepared (marshal-once) batched calls give the bits of the direct calls.

encode_multi_prepared / decode_multi_prepared marshal the job array once and
only make the C call afterwards; the records and rows they produce must equal
those of encode_multi / decode_multi on the same jobs, call after call.
"""
import pytest

import workloads

pytestmark = pytest.mark.gpu


def test_prepared_encode_decode_match_direct(tac_gpu):
    import torch
    tac = tac_gpu
    w = workloads.CONFIGS["mistral7b"]
    enc, dec, xs = [], [], []
    for layer, kv, (n, b, mode) in ((0, 0, (256, 8, 0)), (5, 1, (64, 4, 1)), (7, 0, (56, 32, 2))):
        cfg = tac.layer_cfg(128, n, b, mode, 0, layer, kv)
        x = workloads.block(w, layer, kv, tokens=40, device="cuda")          # 320 rows, ragged tail tile
        cache = tac.Cache.empty(cfg, x.shape[0], device="cuda")
        y = torch.empty_like(x)
        enc.append(tac.EncodeJob(cfg, x, cache))
        dec.append(tac.DecodeJob(cfg, cache, y))
        xs.append(x)
    tac.encode_multi(enc)
    tac.decode_multi(dec)
    torch.cuda.synchronize()
    want_rec = [(j.cache.codes.clone(), j.cache.norms.clone()) for j in enc]
    want_y = [j.y.clone() for j in dec]
    ecall, dcall = tac.encode_multi_prepared(enc), tac.decode_multi_prepared(dec)
    for _ in range(2):
        for j in enc:
            j.cache.codes.zero_()
            j.cache.norms.zero_()
        for j in dec:
            j.y.zero_()
        ecall()
        dcall()
        torch.cuda.synchronize()
        for j, (c, nr) in zip(enc, want_rec):
            assert torch.equal(j.cache.codes, c) and torch.equal(j.cache.norms, nr)
        for j, y in zip(dec, want_y):
            assert torch.equal(j.y, y)
