"""Seeded synthetic KV-cache workloads shaped like the paper's evaluation models.

Inputs only: shapes, value distributions, codebook schedules and record-slot
maps.  Nothing here performs TurboAngle arithmetic (no transform, angle, norm
or packing step); the CUDA path and the CPU oracle both receive these tensors.

The paper measures real KV caches of seven models on WikiText-2 (Sec. 4.1);
neither the weights nor the dataset are available, so these seeded synthetic
caches stand in for them with the same shapes (layers x KV heads x tokens x d)
and the statistical structure the method cares about:

    x[l, kv, h, t, j] = g * sigma[l, kv, h, j] * tau[l, kv, t],   g ~ N(0, 1)

    sigma ~ lognormal(0, s) per channel; exactly max(1, round(p d)) channels per
            (l, kv, h) are outliers, multiplied by m (channel-dependent scales
            and outliers, Sec. 1)
    tau   ~ lognormal(0, s_tok) per token (1 when s_tok = 0)

Every draw is made from numpy/torch generators seeded by (seed, config, layer,
kv) so any block can be regenerated independently.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

K, V = 0, 1
NORM_LINEAR, NORM_LOG, NORM_FP32 = 0, 1, 2


@dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    heads: int
    tokens: int
    d: int
    dtype: str            # "bf16" or "fp32"
    s: float              # channel-scale lognormal sigma
    p: float              # outlier channel fraction
    m: float              # outlier multiplier
    s_tok: float          # per-token lognormal sigma (0 = none)
    n_k: tuple            # per-layer angle bins for K
    n_v: tuple            # per-layer angle bins for V
    b_k: int = 8          # K norms: 8-bit linear (Sec. 3.3, K8V4-log)
    mode_k: int = NORM_LINEAR
    b_v: int = 4          # V norms: 4-bit log-space
    mode_v: int = NORM_LOG

    @property
    def rows_per_block(self) -> int:
        return self.heads * self.tokens

    def codebook(self, layer: int, kv: int):
        """(d, n, norm_bits, norm_mode) of one (layer, K/V) cache."""
        if kv == K:
            return self.d, self.n_k[layer], self.b_k, self.mode_k
        return self.d, self.n_v[layer], self.b_v, self.mode_v

    def blocks(self):
        return [(l, kv) for l in range(self.layers) for kv in (K, V)]


def _boost(L, first, n_early, base):
    n_k = tuple(n_early[0] if l < first else base[0] for l in range(L))
    n_v = tuple(n_early[1] if l < first else base[1] for l in range(L))
    return n_k, n_v


def _make_configs():
    cfgs = {}
    # 1. Tiny single layer: K, V fp32 [8, 1024, 64], n_K = n_V = 64.
    cfgs["tiny"] = Workload("tiny", 1, 8, 1024, 64, "fp32", 0.5, 0.02, 10.0, 0.0, (64,), (64,))
    # 2. Llama-3.2-1B-shaped: 16 L x 8 h x d 64, T 8192, bf16, per-token scale;
    #    layers 0-3 at 256/256, the rest K128/V64.
    nk, nv = _boost(16, 4, (256, 256), (128, 64))
    cfgs["llama1b"] = Workload("llama1b", 16, 8, 8192, 64, "bf16", 0.5, 0.02, 10.0, 0.3, nk, nv)
    # 3. Mistral-7B-shaped: 32 L x 8 h x d 128, T 32768, bf16, lognormal(0,1)
    #    scales, 1% outliers x20; layers 0-3 at n = 256, the rest n = 64.
    nk, nv = _boost(32, 4, (256, 256), (64, 64))
    cfgs["mistral7b"] = Workload("mistral7b", 32, 8, 32768, 128, "bf16", 1.0, 0.01, 20.0, 0.0, nk, nv)
    # 5. Long-context decode sweep: 28 L x 4 h x d 128, T 131072 (codebooks swept).
    cfgs["longctx"] = Workload("longctx", 28, 4, 131072, 128, "bf16", 1.0, 0.01, 20.0, 0.0,
                               (64,) * 28, (64,) * 28)
    # Paper variants (Sec. 3.1 / 3.3, Tables 1-5) on the same value model:
    #  - Mistral-7B angle-only: fp32 pair norms, early-boost (256, 128) on layers
    #    0-3 and the K128/V64 baseline elsewhere (Table 3's Mistral row);
    nk, nv = _boost(32, 4, (256, 128), (128, 64))
    cfgs["mistral7b_angle"] = Workload("mistral7b_angle", 32, 8, 32768, 128, "bf16", 1.0, 0.01, 20.0, 0.0,
                                       nk, nv, 32, NORM_FP32, 32, NORM_FP32)
    #  - Mistral-7B norm8: 8-bit linear norms for K and V (Table 5), codebooks of config 3;
    nk, nv = _boost(32, 4, (256, 256), (64, 64))
    cfgs["mistral7b_norm8"] = Workload("mistral7b_norm8", 32, 8, 32768, 128, "bf16", 1.0, 0.01, 20.0, 0.0,
                                       nk, nv, 8, NORM_LINEAR, 8, NORM_LINEAR)
    #  - TinyLlama-shaped (22 L x 4 KV heads x d 64) with the non-power-of-two n = 56
    #    of Table 1 on every layer, fp32 norms.
    cfgs["tinyllama_n56"] = Workload("tinyllama_n56", 22, 4, 32768, 64, "bf16", 0.5, 0.02, 10.0, 0.0,
                                     (56,) * 22, (56,) * 22, 32, NORM_FP32, 32, NORM_FP32)
    return cfgs


CONFIGS = _make_configs()
# 4. Decode-step append: 256 sequences x 32 L x 8 h x d 128, one token each,
#    codebooks and values as the Mistral-7B config; lengths ~ U[1k, 32k].
APPEND = dict(seqs=256, base="mistral7b", len_lo=1024, len_hi=32768, page=256, pool_pages=256)
SWEEP_N = (16, 32, 64, 128, 256)


def _rng(seed: int, *key) -> np.random.Generator:
    return np.random.default_rng([seed & 0xFFFFFFFF, *[int(k) & 0xFFFFFFFF for k in key]])


def _name_id(name: str) -> int:
    return sum((i + 1) * ord(c) for i, c in enumerate(name)) & 0xFFFF


def channel_scales(w: Workload, layer: int, kv: int, seed: int = 0) -> np.ndarray:
    """sigma[h, j] for one (layer, kv): float64 [heads, d]."""
    g = _rng(seed, _name_id(w.name), 1, layer, kv)
    sig = np.exp(g.normal(0.0, w.s, size=(w.heads, w.d)))
    n_out = max(1, int(round(w.p * w.d)))
    for h in range(w.heads):
        idx = g.choice(w.d, size=n_out, replace=False)
        sig[h, idx] *= w.m
    return sig


def token_scales(w: Workload, layer: int, kv: int, tokens: int | None = None, seed: int = 0):
    """tau[t] for one (layer, kv) (None when the config has no token scale)."""
    if w.s_tok <= 0:
        return None
    g = _rng(seed, _name_id(w.name), 2, layer, kv)
    return np.exp(g.normal(0.0, w.s_tok, size=(tokens or w.tokens,)))


def block(w: Workload, layer: int, kv: int, tokens: int | None = None, seed: int = 0,
          device="cpu", dtype=None):
    """Rows of one (layer, kv) cache as a torch tensor [heads * tokens, d] (row = h*T + t).

    g is drawn with a torch generator on `device` seeded by (seed, config,
    layer, kv), then scaled and rounded to the config dtype (bf16 or fp32).
    """
    import torch
    T = tokens or w.tokens
    sig = torch.tensor(channel_scales(w, layer, kv, seed), dtype=torch.float32, device=device)
    gen = torch.Generator(device=device)
    gen.manual_seed((seed * 1_000_003 + _name_id(w.name) * 7919 + layer * 2 + kv) & 0x7FFFFFFF)
    x = torch.randn((w.heads, T, w.d), generator=gen, device=device, dtype=torch.float32)
    x.mul_(sig[:, None, :])
    tau = token_scales(w, layer, kv, T, seed)
    if tau is not None:
        x.mul_(torch.tensor(tau, dtype=torch.float32, device=device)[None, :, None])
    if dtype is None:
        dtype = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    return x.reshape(w.heads * T, w.d).to(dtype)


def iid_gaussian_rows(rows: int, d: int, seed: int = 0) -> np.ndarray:
    """float64 [rows, d] i.i.d. N(0, 1) (for the uniformity pins)."""
    return _rng(seed, 7, rows, d).standard_normal((rows, d))


def scaled_gaussian_rows(rows: int, d: int, sigma: np.ndarray, seed: int = 0) -> np.ndarray:
    """float64 [rows, d]: N(0, 1) times a fixed channel-scale vector."""
    return _rng(seed, 8, rows, d).standard_normal((rows, d)) * sigma[None, :]


def append_step(seed: int = 0, step: int = 0):
    """Decode-step streaming append (config 4).

    Returns (lengths [seqs], page_of_seq [seqs]): each sequence's current length
    (the position its new token takes) and the physical pool page holding that
    position.  Record slot of (seq s, head h) in each (layer, kv) pool:
        (page_of_seq[s] * heads + h) * page + lengths[s] % page
    so one step writes every row to a scattered slot of a pool of
    pool_pages * heads * page records per (layer, kv).
    """
    a = APPEND
    g = _rng(seed, 4, step)
    lengths = g.integers(a["len_lo"], a["len_hi"] + 1, size=a["seqs"])
    pages = g.permutation(a["pool_pages"])[: a["seqs"]]
    return lengths, pages


def append_slots(seed: int = 0, step: int = 0) -> np.ndarray:
    """int64 [seqs * heads] record slots for the append rows (row = s * heads + h)."""
    a = APPEND
    w = CONFIGS[a["base"]]
    lengths, pages = append_step(seed, step)
    s = np.arange(a["seqs"])[:, None]
    h = np.arange(w.heads)[None, :]
    slots = (pages[s] * w.heads + h) * a["page"] + (lengths[s] % a["page"])
    return slots.reshape(-1).astype(np.int64)


def append_capacity() -> int:
    a = APPEND
    return a["pool_pages"] * CONFIGS[a["base"]].heads * a["page"]
