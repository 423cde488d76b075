"""TurboAngle CPU oracle (arXiv 2603.27467) -- TEST INFRASTRUCTURE ONLY.

Thin ctypes wrapper over ``tac_oracle.c``: a plain, slow fp64 restatement of
the paper's encode/decode path (dense Hadamard, no butterfly).  Only
``tests/``, ``__graft_entry__.smoke()`` and ``bench.py`` (CPU-baseline and
reference legs) may import this package; the product library never does and
shares no code with it.

Every function names the paper passage it restates (section / equation /
algorithm); the C file lists the readings taken where the paper is silent.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tac_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "libtac_oracle.so")
_lib = None
_lock = threading.Lock()

NORM_LINEAR = 0
NORM_LOG = 1


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no FMA contraction, so x86 and Arm agree)."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_SO)
            and os.path.getmtime(_SO) >= os.path.getmtime(_SRC)):
        return _SO
    tmp = _SO + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=gnu11", "-fPIC", "-shared", "-ffp-contract=off",
           "-fno-fast-math", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        c_i64, c_int, c_dbl = ctypes.c_int64, ctypes.c_int, ctypes.c_double
        vp = ctypes.c_void_p
        lib.orc_splitmix64.restype = ctypes.c_uint64
        lib.orc_splitmix64.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
        lib.orc_signs.restype = None
        lib.orc_signs.argtypes = [ctypes.c_uint64, c_int, c_int, c_int, c_int, vp]
        lib.orc_hadamard.restype = None
        lib.orc_hadamard.argtypes = [c_int, vp]
        lib.orc_transform.restype = c_int
        lib.orc_transform.argtypes = [vp, c_i64, c_int, vp, vp]
        lib.orc_encode.restype = c_int
        lib.orc_encode.argtypes = [vp, c_i64, c_int, vp, c_int, c_int, c_int,
                                   vp, vp, vp, vp, vp, vp]
        lib.orc_decode.restype = c_int
        lib.orc_decode.argtypes = [vp, vp, vp, c_i64, c_int, vp, c_int, c_int, c_int, vp]
        lib.orc_pack.restype = c_int
        lib.orc_pack.argtypes = [vp, c_i64, c_int, c_int, vp]
        lib.orc_unpack.restype = c_int
        lib.orc_unpack.argtypes = [vp, c_i64, c_int, c_int, vp]
        lib.orc_slot_pair.restype = c_int
        lib.orc_slot_pair.argtypes = [c_int, c_int]
        lib.orc_pack_record.restype = c_int
        lib.orc_pack_record.argtypes = [vp, c_i64, c_int, c_int, vp]
        lib.orc_unpack_record.restype = c_int
        lib.orc_unpack_record.argtypes = [vp, c_i64, c_int, c_int, vp]
        lib.orc_avg_angle_bits.restype = c_dbl
        lib.orc_avg_angle_bits.argtypes = [c_int, vp, vp]
        lib.orc_total_bits.restype = c_dbl
        lib.orc_total_bits.argtypes = [c_dbl, c_dbl, c_int]
        lib.orc_attend.restype = c_int
        lib.orc_attend.argtypes = [vp, c_int, vp, vp, c_i64, c_int, c_dbl, vp]
        _lib = lib
        return lib


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def splitmix64(seed: int, i: int) -> int:
    """Output #i of SplitMix64 seeded with ``seed`` (used for D, Sec. 2)."""
    return int(_load().orc_splitmix64(seed & (2**64 - 1), i))


def signs(seed: int, layer: int, kv: int, d: int, shared: bool = False) -> np.ndarray:
    """The +-1 diagonal D of Sec. 2 for one (layer, K/V): int8 array of length d."""
    s = np.empty(d, dtype=np.int8)
    _load().orc_signs(seed & (2**64 - 1), layer, kv, int(shared), d, _ptr(s))
    return s


def hadamard(d: int) -> np.ndarray:
    """Normalized Sylvester Hadamard matrix (Sec. 2), d x d float64."""
    H = np.empty((d, d), dtype=np.float64)
    _load().orc_hadamard(d, _ptr(H))
    return H


def transform(x: np.ndarray, s: np.ndarray) -> np.ndarray:
    """y = H D x for each row (Alg. 1, first step)."""
    x = np.ascontiguousarray(x, dtype=np.float64)
    rows, d = x.shape
    y = np.empty_like(x)
    s = np.ascontiguousarray(s, dtype=np.int8)
    rc = _load().orc_transform(_ptr(x), rows, d, _ptr(s), _ptr(y))
    if rc:
        raise ValueError(f"orc_transform failed ({rc})")
    return y


def encode(x: np.ndarray, s: np.ndarray, n: int, b: int, mode: int,
           diagnostics: bool = True) -> dict:
    """Alg. 1 + Eq. 2 (linear or log-space) for every row of x (rows x d, float64).

    Returns dict with k (angle indices), c (norm codes), hdr (stored fp32
    r_min, r_max) and, with ``diagnostics``, edge (distance of theta to the
    nearest bin edge, rad), pre (Eq. 2 pre-round value) and r (exact norms).
    """
    x = np.ascontiguousarray(x, dtype=np.float64)
    rows, d = x.shape
    P = d // 2
    s = np.ascontiguousarray(s, dtype=np.int8)
    k = np.empty((rows, P), dtype=np.int32)
    c = np.empty((rows, P), dtype=np.int32)
    hdr = np.empty((rows, 2), dtype=np.float32)
    edge = np.empty((rows, P), dtype=np.float64) if diagnostics else None
    pre = np.empty((rows, P), dtype=np.float64) if diagnostics else None
    r = np.empty((rows, P), dtype=np.float64) if diagnostics else None
    nul = ctypes.c_void_p(0)
    rc = _load().orc_encode(_ptr(x), rows, d, _ptr(s), n, b, mode, _ptr(k), _ptr(c), _ptr(hdr),
                            _ptr(edge) if diagnostics else nul,
                            _ptr(pre) if diagnostics else nul,
                            _ptr(r) if diagnostics else nul)
    if rc:
        raise ValueError(f"orc_encode failed ({rc})")
    out = {"k": k, "c": c, "hdr": hdr}
    if diagnostics:
        out.update(edge=edge, pre=pre, r=r)
    return out


def decode(k: np.ndarray, c: np.ndarray, hdr: np.ndarray, s: np.ndarray, n: int, b: int,
           mode: int) -> np.ndarray:
    """Sec. 3.1 reconstruction x^ = D H y^ with dequantized norms; float64 rows x d."""
    k = np.ascontiguousarray(k, dtype=np.int32)
    c = np.ascontiguousarray(c, dtype=np.int32)
    hdr = np.ascontiguousarray(hdr, dtype=np.float32)
    rows, P = k.shape
    d = 2 * P
    s = np.ascontiguousarray(s, dtype=np.int8)
    y = np.empty((rows, d), dtype=np.float64)
    rc = _load().orc_decode(_ptr(k), _ptr(c), _ptr(hdr), rows, d, _ptr(s), n, b, mode, _ptr(y))
    if rc:
        raise ValueError(f"orc_decode failed ({rc})")
    return y


def pack(codes: np.ndarray, bits: int) -> np.ndarray:
    """LSB-first dense bit-packing of each row (reading R9); uint8 rows x stride."""
    codes = np.ascontiguousarray(codes, dtype=np.int32)
    rows, count = codes.shape
    stride = (count * bits + 7) // 8
    out = np.empty((rows, stride), dtype=np.uint8)
    if _load().orc_pack(_ptr(codes), rows, count, bits, _ptr(out)):
        raise ValueError("orc_pack failed")
    return out


def unpack(buf: np.ndarray, count: int, bits: int) -> np.ndarray:
    buf = np.ascontiguousarray(buf, dtype=np.uint8)
    rows = buf.shape[0]
    out = np.empty((rows, count), dtype=np.int32)
    if _load().orc_unpack(_ptr(buf), rows, count, bits, _ptr(out)):
        raise ValueError("orc_unpack failed")
    return out


def slot_order(d: int) -> np.ndarray:
    """Record order (reading R9): element v = the pair whose code sits in slot v."""
    lib = _load()
    return np.array([lib.orc_slot_pair(d, v) for v in range(d // 2)], dtype=np.int64)


def pack_record(codes: np.ndarray, d: int, bits: int) -> np.ndarray:
    """Records of rows of d/2 codes given in pair order (slot order, then packed)."""
    codes = np.ascontiguousarray(codes, dtype=np.int32)
    rows = codes.shape[0]
    stride = ((d // 2) * bits + 7) // 8
    out = np.zeros((rows, stride), dtype=np.uint8)
    if _load().orc_pack_record(_ptr(codes), rows, d, bits, _ptr(out)):
        raise ValueError("orc_pack_record failed")
    return out


def unpack_record(buf: np.ndarray, d: int, bits: int) -> np.ndarray:
    """Codes in pair order from records (inverse of pack_record)."""
    buf = np.ascontiguousarray(buf, dtype=np.uint8)
    rows = buf.shape[0]
    out = np.zeros((rows, d // 2), dtype=np.int32)
    if _load().orc_unpack_record(_ptr(buf), rows, d, bits, _ptr(out)):
        raise ValueError("orc_unpack_record failed")
    return out


def avg_angle_bits(nK, nV) -> float:
    """Eq. 1: (1/L) sum_l (log2 n_K + log2 n_V) / 4."""
    a = np.ascontiguousarray(nK, dtype=np.int32)
    b = np.ascontiguousarray(nV, dtype=np.int32)
    return float(_load().orc_avg_angle_bits(len(a), _ptr(a), _ptr(b)))


def total_bits(b_angle: float, b_norm: float, d: int) -> float:
    """Eq. 3: b_angle + b_norm / 2 + 64 / d."""
    return float(_load().orc_total_bits(b_angle, b_norm, d))


def attend(q: np.ndarray, khat: np.ndarray, vhat: np.ndarray, scale: float) -> np.ndarray:
    """Softmax attention of q (nq x d) over decoded rows khat, vhat (T x d), fp64."""
    q = np.ascontiguousarray(q, dtype=np.float64)
    khat = np.ascontiguousarray(khat, dtype=np.float64)
    vhat = np.ascontiguousarray(vhat, dtype=np.float64)
    nq, d = q.shape
    out = np.empty((nq, d), dtype=np.float64)
    if _load().orc_attend(_ptr(q), nq, _ptr(khat), _ptr(vhat), khat.shape[0], d, float(scale), _ptr(out)):
        raise ValueError("orc_attend failed")
    return out


def encode_threads(x: np.ndarray, s: np.ndarray, n: int, b: int, mode: int,
                   threads: int, diagnostics: bool = False) -> dict:
    """encode() over row blocks on ``threads`` host threads (ctypes drops the GIL).

    The per-row arithmetic is exactly encode()'s; only rows are split.  With
    diagnostics the edge distances, pre-round Eq. 2 values and exact norms come
    back too, as from encode().
    """
    x = np.ascontiguousarray(x, dtype=np.float64)
    rows = x.shape[0]
    parts = np.array_split(np.arange(rows), max(1, threads))
    res = [None] * len(parts)

    def work(i, idx):
        if len(idx):
            res[i] = encode(x[idx[0]:idx[-1] + 1], s, n, b, mode, diagnostics=diagnostics)

    ts = [threading.Thread(target=work, args=(i, p)) for i, p in enumerate(parts)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    res = [r for r in res if r is not None]
    return {key: np.concatenate([r[key] for r in res]) for key in res[0]}


def decode_threads(k, c, hdr, s, n, b, mode, threads: int) -> np.ndarray:
    rows = k.shape[0]
    parts = np.array_split(np.arange(rows), max(1, threads))
    res = [None] * len(parts)

    def work(i, idx):
        if len(idx):
            sl = slice(idx[0], idx[-1] + 1)
            res[i] = decode(k[sl], c[sl], hdr[sl], s, n, b, mode)

    ts = [threading.Thread(target=work, args=(i, p)) for i, p in enumerate(parts)]
    for t in ts:
        t.start()
    for t in ts:
        t.join()
    return np.concatenate([r for r in res if r is not None])
