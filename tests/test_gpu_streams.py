"""Batched calls with several kernel shapes run their launches concurrently on
the caller's stream and helper streams joined back by events.

The call must still be ordered on the caller's stream (work queued after it on
that stream sees its results) and must be capturable into a CUDA graph once the
helper streams exist.  Reference results come from the same calls with a device
synchronization after each.
"""
import pytest

import workloads

pytestmark = pytest.mark.gpu


def _jobs(tac):
    import torch
    w = workloads.CONFIGS["mistral7b"]
    enc, dec = [], []
    # four kernel shapes: K/V x base/boosted codebooks, plus a d = 64 job
    specs = [(0, 0, 128, (256, 8, 0)), (0, 1, 128, (256, 4, 1)), (9, 0, 128, (64, 8, 0)),
             (9, 1, 128, (64, 4, 1)), (3, 0, 64, (128, 8, 0))]
    for layer, kv, d, (n, b, mode) in specs:
        cfg = tac.layer_cfg(d, n, b, mode, 0, layer, kv)
        src = workloads.CONFIGS["mistral7b" if d == 128 else "llama1b"]
        x = workloads.block(src, layer, kv, tokens=96, device="cuda")
        cache = tac.Cache.empty(cfg, x.shape[0], device="cuda")
        enc.append(tac.EncodeJob(cfg, x, cache))
        dec.append(tac.DecodeJob(cfg, cache, torch.empty_like(x)))
    return enc, dec


def _reference(tac, enc, dec):
    import torch
    tac.encode_multi(enc)
    torch.cuda.synchronize()
    tac.decode_multi(dec)
    torch.cuda.synchronize()
    return [j.cache.codes.clone() for j in enc], [j.y.clone() for j in dec]


def test_multi_calls_ordered_on_caller_stream(tac_gpu):
    import torch
    tac = tac_gpu
    enc, dec = _jobs(tac)
    want_codes, want_y = _reference(tac, enc, dec)
    s = torch.cuda.Stream()
    for j in enc:
        j.cache.codes.zero_()
    for j in dec:
        j.y.zero_()
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        tac.encode_multi(enc, stream=s)
        codes = [j.cache.codes.clone() for j in enc]     # queued on s right after the call
        tac.decode_multi(dec, stream=s)
        ys = [j.y.clone() for j in dec]
    s.synchronize()
    for a, b in zip(codes, want_codes):
        assert torch.equal(a, b)
    for a, b in zip(ys, want_y):
        assert torch.equal(a, b)


def test_multi_calls_capture_into_graph(tac_gpu):
    import torch
    tac = tac_gpu
    enc, dec = _jobs(tac)
    want_codes, want_y = _reference(tac, enc, dec)      # also creates the helper streams
    ecall, dcall = tac.encode_multi_prepared(enc), tac.decode_multi_prepared(dec)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        ecall(torch.cuda.current_stream())
        dcall(torch.cuda.current_stream())
    for j in enc:
        j.cache.codes.zero_()
    for j in dec:
        j.y.zero_()
    torch.cuda.synchronize()
    for _ in range(2):
        g.replay()
        torch.cuda.synchronize()
        for j, b in zip(enc, want_codes):
            assert torch.equal(j.cache.codes, b)
        for j, b in zip(dec, want_y):
            assert torch.equal(j.y, b)
