#!/usr/bin/env python3
"""TurboAngle KV-cache encode/decode benchmark on GB300 (libtac, sm_103a).

One step = encode every (layer, K/V) block of a synthetic KV cache into packed
records (one tac_encode_multi call: one launch per kernel shape, run
concurrently) and decode every record back to bf16 (one tac_decode_multi call).
Default workload: the Mistral-7B-shaped cache
(32 layers x 8 KV heads x 32768 tokens x d 128, bf16; early-boost n = 256 on
layers 0-3, n = 64 elsewhere; K 8-bit linear / V 4-bit log norms).

value = algorithmic bytes moved per step (bf16 rows in + packed records out for
encode, records in + bf16 rows out for decode) / step time, summed over ranks.
Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl tac|reference]
       [--config mistral7b|llama1b|append|longctx|mistral7b_angle|mistral7b_norm8|
                 tinyllama_n56|attend] [--tokens T] [--graph on|off]
       [--no-e2e] [--no-cpu-baseline] [--probe rd]
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import workloads  # noqa: E402

METRIC = "KV encode / decode GB/s (bf16 in/out) on 1 GB300 and % of HBM peak"
UNIT = "GB/s"
FALLBACK_HBM_GBS = 6800.0

# DRAM bytes per encoded/decoded row that ncu counted: dram__bytes_read.sum +
# dram__bytes_write.sum over every launch of one call (encode: the encode and
# fix-up kernels of each shape) of the 8192-token Mistral-7B-shaped case,
# divided by its 4,194,304 rows; the full-size call has the same codebook mix,
# so its traffic is this figure times its rows.  Each figure holds only for the
# kernel sources it was measured on; after any change to them it reads null.
MEASURED_TRAFFIC = {
    "encode": {"sources": ("tac_common.cuh", "tac_encode.cu"), "sha256_16": "b3b3b2c1be57d737",
               "bytes_per_row": 338.776},
    "decode": {"sources": ("tac_common.cuh", "tac_decode.cu"), "sha256_16": "af89c8435cfc002c",
               "bytes_per_row": 305.386},
    "attend": {"sources": ("tac_common.cuh", "tac_attend.cuh", "tac_attend.cu"), "sha256_16": "4e341a7176bc2a95",
               "bytes_per_row": 221.787},
}


def measured_traffic(kernel: str, rows: int):
    """DRAM bytes of one launch over `rows` rows, or None if the kernel changed."""
    import hashlib
    rec = MEASURED_TRAFFIC.get(kernel)
    if rec is None or not rows:
        return None
    h = hashlib.sha256()
    for f in rec["sources"]:
        with open(os.path.join(ROOT, "paper_2603_27467_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest()[:16] != rec["sha256_16"]:
        return None
    return rec["bytes_per_row"] * rows


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["tac", "reference"], default="tac")
    ap.add_argument("--config", default="mistral7b",
                    choices=["mistral7b", "llama1b", "append", "longctx", "mistral7b_angle", "mistral7b_norm8",
                             "tinyllama_n56", "attend"])
    ap.add_argument("--graph", choices=["on", "off"], default="off",
                    help="replay each timed step's calls from a CUDA graph captured once")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=5)
    ap.add_argument("--e2e-chunk", type=int, default=8, help="(layer, K/V) blocks per e2e pipeline chunk")
    ap.add_argument("--tokens", type=int, default=0,
                    help="override tokens per (layer, K/V) block (smaller cases for profiling)")
    ap.add_argument("--probe", choices=["rd"], default=None,
                    help="rd: rate-distortion probe (relative MSE vs n on the workload distributions)")
    ap.add_argument("--cpu-rows", type=int, default=400_000,
                    help="rows in the bounded oracle sample (CPU baseline / reference arm)")
    return ap.parse_args()


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    Q = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.proc = None
        self.lines = []
        self.thread = None

    def start(self):
        try:
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "100"]
            if self.uuid:
                cmd += ["-i", self.uuid]
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=5)
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 10:
                continue
            try:
                sm.append(float(f[2])); smax.append(float(f[3]))
                power.append(float(f[4]))
            except ValueError:
                continue
            for nm, v in zip(names, f[6:10]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# workloads
# ---------------------------------------------------------------------------
def record_bytes(d, n, b, mode=0):
    """Packed record bytes per row: ceil(log2 n)-bit angle codes, b-bit norms and
    the 8-byte (r_min, r_max) header (no header with fp32 norms)."""
    import math
    hdr = 0 if mode == workloads.NORM_FP32 else 8
    return d // 2 * int(math.ceil(math.log2(n))) // 8 + d // 2 * b // 8 + hdr


def config_desc(name):
    if name == "append":
        a = workloads.APPEND
        w = workloads.CONFIGS[a["base"]]
        return (f"decode-step append: {a['seqs']} seqs x {w.layers} L x 2 (K,V) x {w.heads} KV heads x d {w.d}, "
                f"1 bf16 token each into paged pools ({a['pool_pages']} pages x {a['page']} tok per (L,kv)), "
                "codebooks as mistral7b; encode only")
    w = workloads.CONFIGS[name]
    sched = "early-boost" if len(set(w.n_k)) > 1 else "uniform"

    def norms(b, mode):
        return "fp32" if mode == workloads.NORM_FP32 else f"{b}-bit {'log' if mode == workloads.NORM_LOG else 'linear'}"
    return (f"{name}-shaped KV cache: {w.layers} L x 2 (K,V) x {w.heads} KV heads x {w.tokens} T x d {w.d}, "
            f"{w.dtype}; {sched} n_K={sorted(set(w.n_k))} n_V={sorted(set(w.n_v))}; "
            f"K {norms(w.b_k, w.mode_k)} / V {norms(w.b_v, w.mode_v)} norms")


class Workset:
    """Device-resident cache, records and decode output of one rank, plus byte accounting."""

    def __init__(self, tac, name, seed, device, tokens=0):
        import torch
        self.name = name
        self.enc_jobs, self.dec_jobs = [], []
        self.enc_bytes = 0
        self.dec_bytes = 0
        self.tokens = 0
        if name == "append":
            a = workloads.APPEND
            w = workloads.CONFIGS[a["base"]]
            rows = a["seqs"] * w.heads
            blocks = w.blocks()
            self.x_all = torch.empty((len(blocks), rows, w.d), dtype=torch.bfloat16, device=device)
            slots = torch.from_numpy(workloads.append_slots(seed, 0)).to(device)
            cap = workloads.append_capacity()
            for bi, (l, kv) in enumerate(blocks):
                d, n, b, mode = w.codebook(l, kv)
                cfg = tac.layer_cfg(d, n, b, mode, seed, l, kv)
                x = workloads.block(w, l, kv, tokens=a["seqs"], seed=seed + 11, device=device)
                self.x_all[bi].copy_(x.view(w.heads, a["seqs"], d).transpose(0, 1).reshape(rows, d))
                cache = tac.Cache.empty(cfg, cap, device=device)
                self.enc_jobs.append(tac.EncodeJob(cfg, self.x_all[bi], cache, slots))
                self.enc_bytes += rows * (2 * d + record_bytes(d, n, b, mode))
            self.tokens = a["seqs"]
            self.y_all = None
            self.rows_per_launch = None   # scattered single-token rows: no traffic figure
            return
        w = workloads.CONFIGS[name]
        if tokens:
            import dataclasses
            w = dataclasses.replace(w, tokens=tokens)
        blocks = w.blocks()
        R = w.rows_per_block
        self.x_all = torch.empty((len(blocks), R, w.d), dtype=torch.bfloat16, device=device)
        self.y_all = torch.empty_like(self.x_all)
        for bi, (l, kv) in enumerate(blocks):
            d, n, b, mode = w.codebook(l, kv)
            cfg = tac.layer_cfg(d, n, b, mode, seed, l, kv)
            self.x_all[bi].copy_(workloads.block(w, l, kv, seed=seed, device=device, dtype=torch.bfloat16))
            cache = tac.Cache.empty(cfg, R, device=device)
            self.enc_jobs.append(tac.EncodeJob(cfg, self.x_all[bi], cache))
            self.dec_jobs.append(tac.DecodeJob(cfg, cache, self.y_all[bi]))
            rb = record_bytes(d, n, b, mode)
            self.enc_bytes += R * (2 * d + rb)
            self.dec_bytes += R * (rb + 2 * d)
        self.tokens = w.tokens
        # the measured per-row traffic holds for the Mistral-7B-shaped codebook mix
        self.rows_per_launch = R * len(blocks) if name == "mistral7b" else None

    @property
    def step_bytes(self):
        return self.enc_bytes + self.dec_bytes


# ---------------------------------------------------------------------------
# CPU oracle on a bounded sample (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------
def oracle_sample(name, total_rows, seed=0):
    """A bounded sample of the workload: the first rows of every (layer, K/V) block."""
    import numpy as np
    base = workloads.APPEND["base"] if name == "append" else name
    w = workloads.CONFIGS[base]
    blocks = w.blocks()
    per = max(8, total_rows // len(blocks))
    out = []
    for (l, kv) in blocks:
        x = workloads.block(w, l, kv, tokens=-(-per // w.heads), seed=seed)[:per].double().numpy()
        out.append(((l, kv), np.ascontiguousarray(x)))
    return w, out


def run_oracle(w, sample, threads, do_decode=True):
    import oracle
    nbytes = 0
    t0 = time.perf_counter()
    for (l, kv), x in sample:
        d, n, b, mode = w.codebook(l, kv)
        s = oracle.signs(0, l, kv, d)
        r = oracle.encode_threads(x, s, n, b, mode, threads)
        rb = record_bytes(d, n, b, mode)
        nbytes += x.shape[0] * (2 * d + rb)
        if do_decode:
            oracle.decode_threads(r["k"], r["c"], r["hdr"], s, n, b, mode, threads)
            nbytes += x.shape[0] * (rb + 2 * d)
    return nbytes, time.perf_counter() - t0


def cpu_baseline(args):
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    w, sample = oracle_sample(args.config, args.cpu_rows)
    rows = sum(x.shape[0] for _, x in sample)
    nbytes, dt = run_oracle(w, sample, threads, do_decode=args.config != "append")
    what = "encode" if args.config == "append" else "encode+decode"
    return {"value": nbytes / dt / 1e9, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{rows} rows ({len(sample)} blocks x {sample[0][1].shape[0]} first rows), {what}, "
                      f"fp64 dense-Hadamard oracle, {dt:.1f} s wall on {threads} host threads"}


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    if args.config == "attend":
        print(json.dumps({"impl": "reference", "unavailable": "the reference arm times the oracle's encode/decode "
                          "workloads; attention from records has no oracle timing mode"}), flush=True)
        return
    import oracle
    oracle.build()
    threads = os.cpu_count() or 1
    per_step = max(2048, args.cpu_rows // 20)
    w, sample = oracle_sample(args.config, per_step)
    rows = sum(x.shape[0] for _, x in sample)
    do_dec = args.config != "append"
    for _ in range(args.warmup):
        run_oracle(w, sample, threads, do_dec)
    times, nbytes = [], 0
    for _ in range(args.steps):
        nb, dt = run_oracle(w, sample, threads, do_dec)
        times.append(dt)
        nbytes = nb
    tot = sum(times)
    value = nbytes * args.steps / tot / 1e9
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": tot / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": config_desc(args.config), "sample_rows_per_step": rows},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": f"{rows} rows per step (first rows of each of {len(sample)} blocks)"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# multi-rank host logic (weak scaling: every rank runs an independent replica)
# ---------------------------------------------------------------------------
def rank_seed(rank: int) -> int:
    """Each rank encodes/decodes its own cache (independent replica, its own inputs)."""
    return rank


def max_over_ranks(ms: float, world: int, device=None) -> float:
    """Slowest rank's time: the job finishes when every replica has."""
    if world <= 1:
        return float(ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, bytes_per_rank_step: int, steps: int, total_ms: float) -> float:
    """Whole-job GB/s: bytes every rank moved over the slowest rank's time."""
    return world * bytes_per_rank_step * steps / (total_ms / 1e3) / 1e9


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------
def run_e2e(tac, ws, world, dev, steps, chunk_blocks, step_bytes, barrier):
    """End-to-end throughput: H2D of the step's rows, encode + decode, D2H of the
    decoded rows, per chunk of `chunk_blocks` (layer, K/V) blocks; chunk c's
    copy in, compute and copy out run on three streams ordered by events, so the
    two copy directions and the kernels of different chunks overlap."""
    import torch
    nb = ws.x_all.shape[0]
    chunks = [(c, min(nb, c + chunk_blocks)) for c in range(0, nb, chunk_blocks)]
    hx = torch.empty(ws.x_all.shape, dtype=ws.x_all.dtype, pin_memory=True)
    hx.copy_(ws.x_all)
    hy = torch.empty(ws.y_all.shape, dtype=ws.y_all.dtype, pin_memory=True)
    hy.zero_()                                        # host pages in place before timing
    s_in, s_cmp, s_out = (torch.cuda.Stream(device=dev) for _ in range(3))
    ev_in = [torch.cuda.Event() for _ in chunks]    # rows of chunk c are on the device
    ev_cmp = [torch.cuda.Event() for _ in chunks]   # chunk c encoded and decoded
    ev_out = [torch.cuda.Event() for _ in chunks]   # decoded rows of chunk c are on the host
    state = {"first": True}
    enc_calls = [tac.encode_multi_prepared(ws.enc_jobs[lo:hi]) for lo, hi in chunks]
    dec_calls = [tac.decode_multi_prepared(ws.dec_jobs[lo:hi]) for lo, hi in chunks]

    def one_step():
        first = state["first"]
        for c, (lo, hi) in enumerate(chunks):
            with torch.cuda.stream(s_in):
                if not first:
                    s_in.wait_event(ev_cmp[c])        # last step's encode has read these rows
                ws.x_all[lo:hi].copy_(hx[lo:hi], non_blocking=True)
                ev_in[c].record(s_in)
            with torch.cuda.stream(s_cmp):
                s_cmp.wait_event(ev_in[c])
                if not first:
                    s_cmp.wait_event(ev_out[c])       # last step's copy-out has read these rows
                enc_calls[c](s_cmp)
                dec_calls[c](s_cmp)
                ev_cmp[c].record(s_cmp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(ev_cmp[c])
                hy[lo:hi].copy_(ws.y_all[lo:hi], non_blocking=True)
                ev_out[c].record(s_out)
        state["first"] = False

    for _ in range(2):                                # warm-up
        one_step()
    barrier()
    # Nine timed rounds of `steps` steps; the median round is reported (rounds
    # on the shared host alternate between two link rates, about 2.5x apart,
    # listed in round_ms_per_step).
    rounds = []
    for _ in range(9):
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(s_in)
        for _ in range(steps):
            one_step()
        e1.record(s_out)
        barrier()
        rounds.append(max_over_ranks(e0.elapsed_time(e1), world, dev))
    ms = sorted(rounds)[len(rounds) // 2]
    out = {"value": job_throughput(world, step_bytes, steps, ms), "unit": UNIT,
           "h2d_bytes_per_step": hx.numel() * hx.element_size(),
           "d2h_bytes_per_step": hy.numel() * hy.element_size(),
           "ms_per_step": ms / steps,
           "round_ms_per_step": [r / steps for r in rounds],
           "pipeline": f"{len(chunks)} chunks of {chunk_blocks} blocks; copy in / encode+decode / copy out on 3 streams; "
                       f"median of {len(rounds)} rounds of {steps} steps"}
    del hx, hy
    return out


def run_attend(args):
    """Attention straight from records (tac_attend_multi) on the Mistral-7B-shaped
    cache: one job per (layer, KV head) over all its tokens, 4 query rows per KV
    head (GQA 4:1), bf16 queries and outputs.  value = record bytes read per
    step (K and V records of every token) / step time."""
    import torch
    from paper_2603_27467_gb300 import build as tb
    tb.build()
    import paper_2603_27467_gb300 as tac
    tac.load()
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    w = workloads.CONFIGS["mistral7b"]
    T = args.tokens or w.tokens
    nq = 4
    jobs, rec_bytes, keep = [], 0, []
    for l in range(w.layers):
        caches = {}
        for kv in (workloads.K, workloads.V):
            d, n, b, mode = w.codebook(l, kv)
            cfg = tac.layer_cfg(d, n, b, mode, 0, l, kv)
            x = workloads.block(w, l, kv, tokens=T, device=dev, dtype=torch.bfloat16)
            per_head = []
            for h in range(w.heads):
                c = tac.Cache.empty(cfg, T, device=dev)
                tac.encode(x[h * T:(h + 1) * T], cfg, cache=c)
                per_head.append(c)
            caches[kv] = (cfg, per_head, record_bytes(d, n, b, mode))
            del x
        kcfg, kc, kb = caches[workloads.K]
        vcfg, vc, vb = caches[workloads.V]
        for h in range(w.heads):
            g = torch.Generator(device=dev)
            g.manual_seed(l * 64 + h)
            q = torch.randn((nq, w.d), generator=g, device=dev).to(torch.bfloat16)
            out = torch.empty_like(q)
            jobs.append(tac.AttendJob(kcfg, kc[h], vcfg, vc[h], T, q, out, 1.0 / w.d ** 0.5))
            rec_bytes += T * (kb + vb)
        keep.append(caches)
    ws = torch.empty(tac.attend_workspace_bytes(jobs), dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)
    call = tac.attend_multi_prepared(jobs, ws)
    for _ in range(args.warmup):
        call(stream)
    torch.cuda.synchronize()
    clk = ClockSampler(None)
    clk.start()
    time.sleep(0.3)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        call(stream)
    e1.record(stream)
    torch.cuda.synchronize()
    clocks = clk.stop()
    ms = e0.elapsed_time(e1) / args.steps
    hbm, peak_kind = peaks()
    gbs = rec_bytes / (ms / 1e3) / 1e9
    print(json.dumps({
        "metric": "attention from records GB/s (K+V records read) on 1 GB300", "value": gbs, "unit": "GB/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": {"workload": f"mistral7b-shaped cache, {w.layers} L x {w.heads} KV heads x {T} tokens, "
                               f"{nq} query rows per KV head (GQA 4:1), bf16 q/out, one job per (layer, head)",
                   "record_bytes_per_step": rec_bytes},
        "token_heads_per_s": w.layers * w.heads * T / (ms / 1e3),
        "roofline": {"bound": "hbm", "kernel": "attend_partial + attend_combine", "achieved": gbs, "peak": hbm,
                     "unit": "GB/s", "frac": gbs / hbm, "peak_source": f"{peak_kind} hbm_gbs",
                     "traffic": measured_traffic("attend", w.layers * w.heads * T),
                     "traffic_note": "attend_partial + attend_combine DRAM bytes per token-head (all launches of "
                                     "a step) from ncu at 4096 tokens, scaled by token-heads; null once the kernel "
                                     "source changes"},
        "gpu_launches": 2 * args.steps * (1 + (len(jobs) - 1) // tac.ATTEND_MAX_JOBS), "clocks": clocks}), flush=True)


def probe_rd(args):
    """Rate-distortion probe: relative reconstruction MSE (sum |x^ - x|^2 / sum |x|^2)
    of GPU encode -> decode with fp32 norms (angle-only) for every supported n,
    on blocks of the workload distributions, next to the uniform-angle law
    2 - 2 sin(pi/n)/(pi/n).  Tests the power-of-two aliasing conjecture (n = 56
    vs 64) and the effect of the non-uniform angle density of channel-scaled rows."""
    import math
    import torch
    from paper_2603_27467_gb300 import build as tb
    tb.build()
    import paper_2603_27467_gb300 as tac
    tac.load()
    ns = [16, 32, 48, 56, 64, 128, 256]
    out = {}
    for name in ("mistral7b", "llama1b", "tinyllama_n56"):
        w = workloads.CONFIGS[name]
        layers = sorted({0, w.layers // 2, w.layers - 1})
        res = {}
        for n in ns:
            err = tot = 0.0
            for l in layers:
                for kv in (workloads.K, workloads.V):
                    x = workloads.block(w, l, kv, tokens=4096, device="cuda", dtype=torch.bfloat16)
                    cfg = tac.layer_cfg(w.d, n, 32, tac.NORM_FP32, 0, l, kv)
                    y = tac.decode(tac.encode(x, cfg), cfg, dtype=torch.float32)
                    xd = x.double()
                    err += float((y.double() - xd).pow(2).sum())
                    tot += float(xd.pow(2).sum())
            res[str(n)] = err / tot
        out[name] = res
    law = {str(n): 2 - 2 * math.sin(math.pi / n) / (math.pi / n) for n in ns}
    print(json.dumps({"probe": "rate-distortion", "norms": "fp32", "tokens_per_block": 4096,
                      "rel_mse": out, "uniform_angle_law": law}), flush=True)


def main():
    args = parse_args()
    if args.probe == "rd":
        probe_rd(args)
        return
    if args.config == "attend" and args.impl != "reference":
        run_attend(args)
        return
    if args.impl == "reference":
        run_reference(args)
        return
    import torch
    import torch.distributed as dist
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    dev = torch.device("cuda", torch.cuda.current_device())

    from paper_2603_27467_gb300 import build as tb
    tb.build()
    import paper_2603_27467_gb300 as tac
    tac.load()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    ws = Workset(tac, args.config, seed=rank_seed(rank), device=dev, tokens=args.tokens)
    stream = torch.cuda.Stream(device=dev)
    enc_only = args.config == "append"

    enc_call = tac.encode_multi_prepared(ws.enc_jobs)
    dec_call = tac.decode_multi_prepared(ws.dec_jobs)

    def step():
        enc_call(stream)
        if not enc_only:
            dec_call(stream)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    barrier()

    # A serving loop replays a small step from a CUDA graph: the calls are
    # captured once (after the warm-up has created the library's helper streams
    # and set its kernel attributes) and the graphs are replayed on `stream`.
    use_graph = args.graph == "on"
    g_enc = g_dec = None
    if use_graph:
        g_enc = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_enc, stream=stream):
            enc_call(stream)
        if not enc_only:
            g_dec = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_dec, stream=stream):
                dec_call(stream)

    def run_enc():
        if g_enc is None:
            enc_call(stream)
        else:
            with torch.cuda.stream(stream):
                g_enc.replay()

    def run_dec():
        if g_dec is None:
            dec_call(stream)
        else:
            with torch.cuda.stream(stream):
                g_dec.replay()

    if use_graph:
        for _ in range(3):
            run_enc()
            if not enc_only:
                run_dec()
    barrier()

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    uuid = None
    try:
        uuid = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        uuid = None
    # Inputs smaller than twice the L2: flush it between timed steps and time
    # the steps themselves.  The flush writes a buffer of twice the L2's size,
    # then reads another of that size, so that the lines it leaves are clean:
    # the write-back of its own dirty lines happens before the timed step
    # instead of inside it.
    l2 = int(getattr(torch.cuda.get_device_properties(dev), "L2_cache_size", 0) or (129 << 20))
    in_bytes = ws.x_all.numel() * ws.x_all.element_size()
    flush = torch.empty(2 * l2 // 4, dtype=torch.int32, device=dev) if in_bytes < 2 * l2 else None
    flush_r = torch.ones(2 * l2 // 4, dtype=torch.int32, device=dev) if flush is not None else None
    clk = ClockSampler(uuid)
    clk.start()
    time.sleep(0.3)
    barrier()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for i in range(K):
        if flush is not None:
            with torch.cuda.stream(stream):
                flush.fill_(i)
                flush_r.max()
        ev[i][0].record(stream)
        run_enc()
        ev[i][1].record(stream)
        if not enc_only:
            run_dec()
        ev[i][2].record(stream)
    t_end.record(stream)
    barrier()
    clocks = clk.stop()
    total_ms = t_start.elapsed_time(t_end)
    if flush is not None:   # the flushes are outside the timed steps
        total_ms = sum(e[0].elapsed_time(e[2]) for e in ev)
    enc_ms = [e[0].elapsed_time(e[1]) for e in ev]
    dec_ms = [e[1].elapsed_time(e[2]) for e in ev] if not enc_only else [0.0]
    total_ms = max_over_ranks(total_ms, world, dev)
    launches_per_step = tac.launch_count(ws.enc_jobs) + (0 if enc_only else tac.launch_count(ws.dec_jobs))

    step_bytes = ws.enc_bytes + (0 if enc_only else ws.dec_bytes)
    value = job_throughput(world, step_bytes, K, total_ms)
    hbm, peak_kind = peaks()
    enc_avg = statistics.mean(enc_ms)
    dec_avg = statistics.mean(dec_ms)
    enc_gbs = ws.enc_bytes / (enc_avg / 1e3) / 1e9
    dec_gbs = ws.dec_bytes / (dec_avg / 1e3) / 1e9 if not enc_only else None
    dom = "encode" if enc_only or sum(enc_ms) >= sum(dec_ms) else "decode"
    dom_gbs = enc_gbs if dom == "encode" else dec_gbs
    dom_bytes = ws.enc_bytes if dom == "encode" else ws.dec_bytes

    # e2e: the same step through the C ABI from pinned host buffers, with the
    # host->device copy of every step's rows and the device->host read of its
    # decoded rows inside the timed region, pipelined over chunks of blocks on
    # three streams (copy in / encode+decode / copy out).
    e2e = None
    if not args.no_e2e and not enc_only:
        e2e = run_e2e(tac, ws, world, dev, args.e2e_steps, args.e2e_chunk, step_bytes, barrier)

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args)

    if rank == 0:
        w = workloads.CONFIGS[workloads.APPEND["base"] if enc_only else args.config]
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
            "warmup": args.warmup, "ms_per_step": total_ms / K, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": {"workload": config_desc(args.config) + (f" (tokens overridden: {args.tokens})" if args.tokens else ""),
                       "io_dtype": "bf16",
                       "bytes_per_step_per_gpu": step_bytes,
                       "l2": (f"L2 flushed before every timed step ({2 * l2 / 1e6:.0f} MB written, then "
                              f"{2 * l2 / 1e6:.0f} MB of another buffer read, not timed); "
                              f"{in_bytes / 1e6:.1f} MB of bf16 rows per step"
                              if flush is not None else
                              "inputs larger than L2 (no flush needed): "
                              f"{in_bytes / 1e9:.2f} GB of bf16 rows per step"),
                       "parallelism": f"replicas x{world} (independent caches, no collective)",
                       "launch": ("each call replayed from a CUDA graph captured once (launches and stream "
                                  "fork / join inside the graph)" if use_graph else
                                  "direct stream-ordered calls (prepared job arrays)")},
            "pct_hbm_peak": 100.0 * value / world / hbm,
            "encode_gbs": enc_gbs, "decode_gbs": dec_gbs,
            "tokens_per_s": world * ws.tokens * w.layers * K / (total_ms / 1e3),
            "roofline": {"bound": "hbm", "kernel": f"{dom} (one tac_{dom}_multi call: one launch per kernel shape, run concurrently)",
                         "achieved": dom_gbs, "peak": hbm, "unit": "GB/s", "frac": dom_gbs / hbm,
                         "peak_source": f"{peak_kind} hbm_gbs",
                         "traffic": measured_traffic(dom, ws.rows_per_launch),
                         "algorithmic_bytes_per_launch": dom_bytes},
            "cpu_baseline": cpu, "e2e": e2e, "gpu_launches": launches_per_step * K, "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
