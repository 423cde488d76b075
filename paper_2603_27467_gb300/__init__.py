"""libtac Python binding: TurboAngle KV-cache encode/decode on GB300 (arXiv 2603.27467).

Argument marshalling only.  Every step of encode and decode runs in the CUDA
kernels of ``libtac.so`` (C ABI declared in ``include/tac.h``); PyTorch is used
for device memory and streams.  There is no CPU path: if the library is not
built, or no CUDA device is present, calls raise.

Names follow the C ABI: ``make_signs``, ``encode``, ``decode``, ``encode_multi``,
``decode_multi``, ``fwht_debug``, plus the plane-geometry and rate helpers
(Eq. 1 and Eq. 3 of the paper).
"""
from __future__ import annotations

import ctypes
import os
import threading
from dataclasses import dataclass, field

import numpy as np

__all__ = [
    "TAC_OK", "TAC_E_INVAL", "TAC_E_UNSUPPORTED", "TAC_E_CUDA", "TAC_E_NONFINITE", "NORM_LINEAR", "NORM_LOG", "NORM_FP32",
    "BF16", "FP32", "TacError", "LayerCfg", "EncodeJob", "DecodeJob", "library_path", "load",
    "make_signs", "layer_cfg", "angle_row_bytes", "norm_row_bytes", "header_offset",
    "codes_bytes", "norms_bytes", "avg_angle_bits", "total_bits", "encode", "decode",
    "encode_multi", "decode_multi", "fwht_debug", "last_error", "version", "Cache",
    "AttendJob", "attend_multi", "attend_workspace_bytes",
]

TAC_OK, TAC_E_INVAL, TAC_E_UNSUPPORTED, TAC_E_CUDA, TAC_E_NONFINITE = 0, 1, 2, 3, 4
NORM_LINEAR, NORM_LOG, NORM_FP32 = 0, 1, 2
BF16, FP32 = 0, 1
MAX_D = 128
MAX_JOBS = 96  # TAC_MAX_JOBS: jobs per kernel launch
ATTEND_STATIC_WS_BYTES = 8 << 20  # TAC_ATTEND_STATIC_WS_BYTES: static attention workspace per device
ATTEND_MAX_JOBS = 160  # TAC_ATTEND_MAX_JOBS: jobs per attention launch pair

_HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(_HERE, "_build", "libtac.so")
_lib = None
_lock = threading.Lock()


class TacError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"libtac error {code}: {msg}")
        self.code = code


class _Cfg(ctypes.Structure):
    _fields_ = [("d", ctypes.c_int32), ("n_angle", ctypes.c_int32), ("norm_bits", ctypes.c_int32),
                ("norm_mode", ctypes.c_int32), ("signs", ctypes.c_uint32 * (MAX_D // 32))]


class _Rows(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("dtype", ctypes.c_int32), ("rows", ctypes.c_int64),
                ("row_stride", ctypes.c_int64)]


class _EncJob(ctypes.Structure):
    _fields_ = [("cfg", _Cfg), ("x", _Rows), ("codes", ctypes.c_void_p), ("norms", ctypes.c_void_p),
                ("capacity", ctypes.c_int64), ("slot", ctypes.c_void_p), ("status", ctypes.c_void_p)]


class _DecJob(ctypes.Structure):
    _fields_ = [("cfg", _Cfg), ("codes", ctypes.c_void_p), ("norms", ctypes.c_void_p),
                ("capacity", ctypes.c_int64), ("slot", ctypes.c_void_p), ("y", _Rows)]


class _AttJob(ctypes.Structure):
    _fields_ = [("cfg_k", _Cfg), ("cfg_v", _Cfg), ("k_codes", ctypes.c_void_p), ("k_norms", ctypes.c_void_p),
                ("v_codes", ctypes.c_void_p), ("v_norms", ctypes.c_void_p), ("capacity", ctypes.c_int64),
                ("tokens", ctypes.c_int64), ("q", _Rows), ("out", _Rows), ("scale", ctypes.c_float)]


def library_path() -> str:
    return _LIB_PATH


def load():
    """Load libtac.so (raises if it has not been built: there is no fallback)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libtac.so not built ({_LIB_PATH}); run "
                               "`python -c 'import __graft_entry__ as g; g.build()'`")
        lib = ctypes.CDLL(_LIB_PATH)
        i64, i32, vp = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
        P = ctypes.POINTER
        lib.tac_make_signs.restype = i32
        lib.tac_make_signs.argtypes = [ctypes.c_uint64, i32, i32, i32, P(ctypes.c_uint32)]
        lib.tac_make_signs_shared.restype = i32
        lib.tac_make_signs_shared.argtypes = [ctypes.c_uint64, i32, P(ctypes.c_uint32)]
        lib.tac_rates.restype = i32
        lib.tac_rates.argtypes = [i32, P(ctypes.c_int), P(ctypes.c_int), i32, i32, i32, P(ctypes.c_double)]
        for name in ("tac_angle_row_bytes", "tac_norm_row_bytes"):
            getattr(lib, name).restype = i64
            getattr(lib, name).argtypes = [P(_Cfg)]
        for name in ("tac_header_offset", "tac_codes_bytes", "tac_norms_bytes"):
            getattr(lib, name).restype = i64
            getattr(lib, name).argtypes = [P(_Cfg), i64]
        lib.tac_avg_angle_bits.restype = ctypes.c_double
        lib.tac_avg_angle_bits.argtypes = [i32, P(ctypes.c_int), P(ctypes.c_int)]
        lib.tac_total_bits.restype = ctypes.c_double
        lib.tac_total_bits.argtypes = [ctypes.c_double, ctypes.c_double, i32]
        lib.tac_encode.restype = i32
        lib.tac_encode.argtypes = [P(_Rows), P(_Cfg), vp, vp, vp]
        lib.tac_encode_checked.restype = i32
        lib.tac_encode_checked.argtypes = [P(_Rows), P(_Cfg), vp, vp, vp, vp]
        lib.tac_decode.restype = i32
        lib.tac_decode.argtypes = [vp, vp, P(_Cfg), P(_Rows), vp]
        lib.tac_encode_multi.restype = i32
        lib.tac_encode_multi.argtypes = [P(_EncJob), i32, vp]
        lib.tac_encode_workspace_bytes.restype = i64
        lib.tac_encode_workspace_bytes.argtypes = [P(_EncJob), i32, P(ctypes.c_int64)]
        lib.tac_encode_multi_ws.restype = i32
        lib.tac_encode_multi_ws.argtypes = [P(_EncJob), i32, vp, i64, vp]
        lib.tac_decode_multi.restype = i32
        lib.tac_decode_multi.argtypes = [P(_DecJob), i32, vp]
        lib.tac_attend_workspace_bytes.restype = i64
        lib.tac_attend_workspace_bytes.argtypes = [P(_AttJob), i32]
        lib.tac_attend_multi.restype = i32
        lib.tac_attend_multi.argtypes = [P(_AttJob), i32, vp, i64, vp]
        lib.tac_attend_multi_static.restype = i32
        lib.tac_attend_multi_static.argtypes = [P(_AttJob), i32, vp]
        lib.tac_fwht_debug.restype = i32
        lib.tac_fwht_debug.argtypes = [P(_Rows), i32, P(ctypes.c_uint32), vp, vp]
        lib.tac_hw_approx_debug.restype = i32
        lib.tac_hw_approx_debug.argtypes = [i32, vp, vp, i64, vp]
        lib.tac_last_error.restype = ctypes.c_char_p
        lib.tac_last_error.argtypes = []
        lib.tac_version.restype = ctypes.c_char_p
        lib.tac_version.argtypes = []
        _lib = lib
        return lib


def last_error() -> str:
    return load().tac_last_error().decode()


def version() -> str:
    return load().tac_version().decode()


def _check(rc: int):
    if rc != TAC_OK:
        raise TacError(rc, last_error())


# ---------------------------------------------------------------------------
# Codebook configuration (Sec. 3.2 per-layer (n_K, n_V); Sec. 3.3 norm bits/mode)
# ---------------------------------------------------------------------------
@dataclass
class LayerCfg:
    d: int
    n_angle: int
    norm_bits: int
    norm_mode: int
    signs: np.ndarray = field(default_factory=lambda: np.zeros(MAX_D // 32, dtype=np.uint32))

    def to_c(self) -> _Cfg:
        c = _Cfg()
        c.d, c.n_angle, c.norm_bits, c.norm_mode = self.d, self.n_angle, self.norm_bits, self.norm_mode
        s = np.zeros(MAX_D // 32, dtype=np.uint32)
        s[: len(self.signs)] = self.signs
        for q in range(MAX_D // 32):
            c.signs[q] = int(s[q])
        return c


def make_signs(seed: int, layer: int, kv: int, d: int, shared: bool = False) -> np.ndarray:
    """D of Sec. 2 for (layer, kv) as little-endian uint32 bit words (bit set => -1)."""
    words = np.zeros(max(1, (d + 31) // 32), dtype=np.uint32)
    out = words.ctypes.data_as(ctypes.POINTER(ctypes.c_uint32))
    if shared:
        _check(load().tac_make_signs_shared(seed & (2**64 - 1), d, out))
    else:
        _check(load().tac_make_signs(seed & (2**64 - 1), layer, kv, d, out))
    return words


def layer_cfg(d: int, n_angle: int, norm_bits: int, norm_mode: int, seed: int = 0, layer: int = 0,
              kv: int = 0, shared: bool = False) -> LayerCfg:
    return LayerCfg(d, n_angle, norm_bits, norm_mode, make_signs(seed, layer, kv, d, shared))


def _geom(name, cfg: LayerCfg, *args):
    c = cfg.to_c()
    v = getattr(load(), name)(ctypes.byref(c), *args)
    if v < 0:
        raise TacError(TAC_E_INVAL, last_error())
    return int(v)


def angle_row_bytes(cfg: LayerCfg) -> int:
    return _geom("tac_angle_row_bytes", cfg)


def norm_row_bytes(cfg: LayerCfg) -> int:
    return _geom("tac_norm_row_bytes", cfg)


def header_offset(cfg: LayerCfg, capacity: int) -> int:
    return _geom("tac_header_offset", cfg, capacity)


def codes_bytes(cfg: LayerCfg, capacity: int) -> int:
    return _geom("tac_codes_bytes", cfg, capacity)


def norms_bytes(cfg: LayerCfg, capacity: int) -> int:
    return _geom("tac_norms_bytes", cfg, capacity)


def avg_angle_bits(n_k, n_v) -> float:
    """Eq. 1."""
    a = (ctypes.c_int * len(n_k))(*[int(v) for v in n_k])
    b = (ctypes.c_int * len(n_v))(*[int(v) for v in n_v])
    return float(load().tac_avg_angle_bits(len(n_k), a, b))


def total_bits(b_angle: float, b_norm: float, d: int) -> float:
    """Eq. 3."""
    return float(load().tac_total_bits(b_angle, b_norm, d))


# ---------------------------------------------------------------------------
# torch marshalling
# ---------------------------------------------------------------------------
def _torch():
    import torch  # noqa: WPS433 (device memory and streams only)
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return FP32
    raise TypeError(f"unsupported dtype {t.dtype} (bf16 or fp32)")


def _rows(t, d: int) -> _Rows:
    if t.dim() != 2 or t.shape[1] != d or (t.shape[0] > 1 and t.stride(1) != 1):
        raise ValueError(f"expected a [rows, {d}] tensor with unit inner stride, got {tuple(t.shape)}")
    if not t.is_cuda:
        raise ValueError("tensor must be on a CUDA device")
    r = _Rows()
    r.data = t.data_ptr()
    r.dtype = _dtype_code(t)
    r.rows = t.shape[0]
    r.row_stride = t.stride(0) if t.shape[0] > 1 else d
    return r


def _stream_ptr(stream) -> int:
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


@dataclass
class Cache:
    """Record planes of one (layer, K/V) cache: angle plane and norm+header planes."""
    cfg: LayerCfg
    capacity: int
    codes: object  # torch.uint8 device tensor
    norms: object  # torch.uint8 device tensor

    @staticmethod
    def empty(cfg: LayerCfg, capacity: int, device="cuda") -> "Cache":
        torch = _torch()
        cb, nb = codes_bytes(cfg, capacity), norms_bytes(cfg, capacity)
        # 16-byte aligned (the caching allocator returns >= 512-byte aligned blocks)
        codes = torch.empty(max(cb, 16), dtype=torch.uint8, device=device)
        norms = torch.empty(max(nb, 16), dtype=torch.uint8, device=device)
        return Cache(cfg, capacity, codes, norms)

    def planes(self):
        """Host views (numpy) of (angle plane, norm plane, header (r_min, r_max));
        with fp32 norms there is no header plane and the header is None."""
        ab, nb = angle_row_bytes(self.cfg), norm_row_bytes(self.cfg)
        off = header_offset(self.cfg, self.capacity)
        codes = self.codes.cpu().numpy()[: self.capacity * ab].reshape(self.capacity, ab)
        nh = self.norms.cpu().numpy()
        norms = nh[: self.capacity * nb].reshape(self.capacity, nb)
        if self.cfg.norm_mode == NORM_FP32:
            return codes, norms, None
        hdr = nh[off: off + 8 * self.capacity].view(np.float32).reshape(self.capacity, 2)
        return codes, norms, hdr


@dataclass
class EncodeJob:
    cfg: LayerCfg
    x: object            # [rows, d] bf16/fp32 device tensor
    cache: Cache
    slot: object = None  # optional int64 device tensor [rows]
    status: object = None  # optional int32 device tensor [1], zeroed: gets TAC_E_NONFINITE


@dataclass
class DecodeJob:
    cfg: LayerCfg
    cache: Cache
    y: object            # [rows, d] bf16/fp32 device tensor (output)
    slot: object = None  # optional int64 device tensor [rows]


def encode(x, cfg: LayerCfg, cache: Cache | None = None, stream=None, status=None) -> Cache:
    """tac_encode: rows of x -> record slots 0..rows-1 of a cache of capacity rows.
    With `status` (an int32 device tensor of one element, zeroed by the caller)
    tac_encode_checked stores TAC_E_NONFINITE in it if a row holds a NaN or an inf."""
    if cache is None:
        cache = Cache.empty(cfg, x.shape[0], device=x.device)
    if cache.capacity != x.shape[0]:
        raise ValueError("tac_encode writes a cache of capacity rows; use encode_multi for slots")
    r = _rows(x, cfg.d)
    c = cfg.to_c()
    if status is None:
        _check(load().tac_encode(ctypes.byref(r), ctypes.byref(c), cache.codes.data_ptr(),
                                 cache.norms.data_ptr(), _stream_ptr(stream)))
    else:
        _check(load().tac_encode_checked(ctypes.byref(r), ctypes.byref(c), cache.codes.data_ptr(),
                                         cache.norms.data_ptr(), status.data_ptr(), _stream_ptr(stream)))
    return cache


def decode(cache: Cache, cfg: LayerCfg, rows: int | None = None, dtype=None, y=None, stream=None):
    """tac_decode: record slots 0..rows-1 -> [rows, d] (bf16 by default)."""
    torch = _torch()
    rows = cache.capacity if rows is None else rows
    if y is None:
        y = torch.empty((rows, cfg.d), dtype=dtype or torch.bfloat16, device=cache.codes.device)
    if rows != cache.capacity:
        raise ValueError("tac_decode reads a cache of capacity rows; use decode_multi for slots")
    r = _rows(y, cfg.d)
    c = cfg.to_c()
    _check(load().tac_decode(cache.codes.data_ptr(), cache.norms.data_ptr(), ctypes.byref(c),
                             ctypes.byref(r), _stream_ptr(stream)))
    return y


class Prepared:
    """A batched call with its job array marshalled once: calling it makes only
    the C call.  The jobs' tensors must stay allocated (their addresses are in
    the array) and the jobs unchanged while it is used.  A prepared encode or
    attention call reuses one workspace on every call, so its calls must not
    overlap in time: make them on one stream, or order the streams."""

    def __init__(self, fn, arr, n, extra, keep):
        self._fn, self._arr, self._n, self._extra, self._keep = fn, arr, n, extra, keep

    def __call__(self, stream=None) -> None:
        _check(self._fn(self._arr, self._n, *self._extra, _stream_ptr(stream)))


def _enc_array(jobs):
    arr = (_EncJob * max(1, len(jobs)))()
    for i, j in enumerate(jobs):
        e = arr[i]
        e.cfg = j.cfg.to_c()
        e.x = _rows(j.x, j.cfg.d)
        e.codes = j.cache.codes.data_ptr()
        e.norms = j.cache.norms.data_ptr()
        e.capacity = j.cache.capacity
        e.slot = j.slot.data_ptr() if j.slot is not None else None
        e.status = j.status.data_ptr() if j.status is not None else None
    return arr


def encode_workspace_bytes(jobs) -> tuple[int, int]:
    """tac_encode_workspace_bytes: (recommended, minimum) workspace bytes."""
    mn = ctypes.c_int64(0)
    n = load().tac_encode_workspace_bytes(_enc_array(jobs), len(jobs), ctypes.byref(mn))
    if n < 0:
        raise TacError(TAC_E_INVAL, last_error())
    return int(n), int(mn.value)


def _enc_workspace(jobs, workspace):
    if workspace is None:
        need = encode_workspace_bytes(jobs)[0] if jobs else 0
        dev = jobs[0].x.device if jobs else "cuda"
        workspace = _torch().empty(max(need, 16), dtype=_torch().uint8, device=dev)
    return workspace


def encode_multi(jobs, stream=None, workspace=None):
    """tac_encode_multi_ws: one encode launch and one fix-up launch per kernel
    group (see launch_count); allocates the re-decision workspace (torch) when
    none is given.  Returns the workspace."""
    arr = _enc_array(jobs)
    workspace = _enc_workspace(jobs, workspace)
    _check(load().tac_encode_multi_ws(arr, len(jobs), workspace.data_ptr(),
                                      workspace.numel() * workspace.element_size(), _stream_ptr(stream)))
    if stream is not None and jobs:
        workspace.record_stream(stream)   # in use on `stream` until its work is done
    return workspace


def encode_multi_prepared(jobs, workspace=None) -> Prepared:
    """tac_encode_multi_ws over `jobs`, marshalled once (see Prepared), with
    a workspace allocated (torch) once when none is given."""
    workspace = _enc_workspace(jobs, workspace)
    extra = (workspace.data_ptr(), workspace.numel() * workspace.element_size())
    return Prepared(load().tac_encode_multi_ws, _enc_array(jobs), len(jobs), extra, (list(jobs), workspace))


def _dec_array(jobs):
    arr = (_DecJob * max(1, len(jobs)))()
    for i, j in enumerate(jobs):
        e = arr[i]
        e.cfg = j.cfg.to_c()
        e.codes = j.cache.codes.data_ptr()
        e.norms = j.cache.norms.data_ptr()
        e.capacity = j.cache.capacity
        e.slot = j.slot.data_ptr() if j.slot is not None else None
        e.y = _rows(j.y, j.cfg.d)
    return arr


def decode_multi(jobs, stream=None) -> None:
    """tac_decode_multi: one launch per kernel group (see launch_count)."""
    _check(load().tac_decode_multi(_dec_array(jobs), len(jobs), _stream_ptr(stream)))


def decode_multi_prepared(jobs) -> Prepared:
    """tac_decode_multi over `jobs`, marshalled once (see Prepared)."""
    return Prepared(load().tac_decode_multi, _dec_array(jobs), len(jobs), (), list(jobs))


@dataclass
class AttendJob:
    """Attention of q rows over record slots 0..tokens-1 of a K and a V cache."""
    k_cfg: LayerCfg
    k_cache: Cache
    v_cfg: LayerCfg
    v_cache: Cache
    tokens: int
    q: object            # [nq, d] bf16/fp32 device tensor, nq <= 8
    out: object          # [nq, d] device tensor, dtype of q
    scale: float


def _att_array(jobs):
    arr = (_AttJob * max(1, len(jobs)))()
    for i, j in enumerate(jobs):
        a = arr[i]
        a.cfg_k, a.cfg_v = j.k_cfg.to_c(), j.v_cfg.to_c()
        a.k_codes, a.k_norms = j.k_cache.codes.data_ptr(), j.k_cache.norms.data_ptr()
        a.v_codes, a.v_norms = j.v_cache.codes.data_ptr(), j.v_cache.norms.data_ptr()
        a.capacity = min(j.k_cache.capacity, j.v_cache.capacity)
        a.tokens = j.tokens
        a.q = _rows(j.q, j.k_cfg.d)
        a.out = _rows(j.out, j.k_cfg.d)
        a.scale = float(j.scale)
    return arr


def attend_workspace_bytes(jobs) -> int:
    """tac_attend_workspace_bytes."""
    n = load().tac_attend_workspace_bytes(_att_array(jobs), len(jobs))
    if n < 0:
        raise TacError(TAC_E_INVAL, last_error())
    return int(n)


def attend_multi(jobs, workspace=None, stream=None):
    """tac_attend_multi; allocates the workspace (torch) when none is given."""
    torch = _torch()
    arr = _att_array(jobs)
    need = attend_workspace_bytes(jobs) if jobs else 0
    if workspace is None:
        dev = jobs[0].q.device if jobs else "cuda"
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    _check(load().tac_attend_multi(arr, len(jobs), workspace.data_ptr() if jobs else None,
                                   workspace.numel() * workspace.element_size(), _stream_ptr(stream)))
    return workspace


def attend_multi_prepared(jobs, workspace=None, static=False) -> Prepared:
    """tac_attend_multi (or tac_attend_multi_static) over `jobs`, marshalled
    once (see Prepared); allocates the workspace (torch) when none is given."""
    lib = load()
    arr = _att_array(jobs)
    if static:
        return Prepared(lib.tac_attend_multi_static, arr, len(jobs), (), list(jobs))
    torch = _torch()
    need = attend_workspace_bytes(jobs) if jobs else 0
    if workspace is None:
        dev = jobs[0].q.device if jobs else "cuda"
        workspace = torch.empty(max(need, 16), dtype=torch.uint8, device=dev)
    extra = (workspace.data_ptr() if jobs else None, workspace.numel() * workspace.element_size())
    return Prepared(lib.tac_attend_multi, arr, len(jobs), extra, (list(jobs), workspace))


def attend_multi_static(jobs, stream=None):
    """tac_attend_multi_static: the library's static device workspace
    (ATTEND_STATIC_WS_BYTES per device), nothing allocated.  An empty job
    list only resolves the workspace address on the current device."""
    _check(load().tac_attend_multi_static(_att_array(jobs), len(jobs), _stream_ptr(stream)))


def launch_count(jobs) -> int:
    """Kernel launches one encode_multi / decode_multi call makes for `jobs`:
    jobs with rows are grouped by kernel (d, dtype, n, norm bits, norm mode),
    at most MAX_JOBS jobs per group; a decode group is one launch, an encode
    group two (the encode and its fix-up)."""
    groups: dict = {}
    per = 1
    for j in jobs:
        t = j.x if isinstance(j, EncodeJob) else j.y
        if isinstance(j, EncodeJob):
            per = 2
        if t.shape[0] == 0:
            continue
        key = (j.cfg.d, str(t.dtype), j.cfg.n_angle, j.cfg.norm_bits, j.cfg.norm_mode)
        groups[key] = groups.get(key, 0) + 1
    return per * sum(-(-c // MAX_JOBS) for c in groups.values())


def fwht_debug(x, signs: np.ndarray, d: int, stream=None):
    """tac_fwht_debug: y = H D x (normalized), fp32 [rows, d]."""
    torch = _torch()
    y = torch.empty((x.shape[0], d), dtype=torch.float32, device=x.device)
    r = _rows(x, d)
    s = (ctypes.c_uint32 * 4)(*([int(v) for v in signs] + [0] * (4 - len(signs))))
    _check(load().tac_fwht_debug(ctypes.byref(r), d, s, y.data_ptr(), _stream_ptr(stream)))
    return y


HW_SQRT, HW_SQRT_FTZ, HW_RCP_FTZ, HW_LG2, HW_LG2_FTZ, HW_EX2_FTZ = range(6)


def hw_approx_debug(op: int, x, stream=None):
    """tac_hw_approx_debug: the kernels' hardware approximation `op` applied to
    the fp32 device tensor x, element-wise."""
    torch = _torch()
    x = x.contiguous()
    y = torch.empty_like(x)
    _check(load().tac_hw_approx_debug(op, x.data_ptr(), y.data_ptr(), x.numel(), _stream_ptr(stream)))
    return y


def rates(d: int, n_k, n_v, b_k: int = 8, b_v: int = 4) -> dict:
    """tac_rates: Eq. 1 angle bits, payload bits (angle + norm bits per pair / 2),
    Eq. 3 total (no min/max header with fp32 norms, b_k = b_v = 32) and the
    ceil(log2 n) bits the angle codes occupy, for a per-layer schedule."""
    L = len(n_k)
    a = (ctypes.c_int * L)(*[int(v) for v in n_k])
    b = (ctypes.c_int * L)(*[int(v) for v in n_v])
    out = (ctypes.c_double * 4)()
    _check(load().tac_rates(L, a, b, b_k, b_v, d, out))
    return {"angle_bits": out[0], "payload_bits": out[1], "total_bits": out[2], "stored_angle_bits": out[3]}


def early_boost(num_layers: int, boosted, n_early=(256, 128), base=(128, 64)):
    """Per-layer MixedKV schedule (Sec. 3.2): (n_K, n_V) = n_early on `boosted`
    layers (an int n_early for layers 0..n-1, or an iterable of layer ids), base elsewhere."""
    if isinstance(boosted, int):
        boosted = range(boosted)
    boosted = set(boosted)
    n_k = [n_early[0] if l in boosted else base[0] for l in range(num_layers)]
    n_v = [n_early[1] if l in boosted else base[1] for l in range(num_layers)]
    return n_k, n_v


__all__ += ["rates", "early_boost"]
