"""Thin Python binding of libris (include/ris.h): argument marshalling only.

Every function has the name of the C entry point it calls and takes torch tensors that are
already on the GPU; all compute runs in the library's CUDA kernels. There is no fallback:
if ``libris.so`` is missing or no CUDA device is present the call raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libris.so")
_lock = threading.Lock()
_lib = None

RIS_OK, RIS_ERR_INVALID, RIS_ERR_OOM, RIS_ERR_CUDA, RIS_ERR_UNSUPPORTED, RIS_ERR_DEVICE_TIMEOUT = range(6)
MODE_STOCHASTIC, MODE_STRUCTURAL, MODE_DENSE = 0, 1, 2
F32, BF16 = 0, 1
ROPE_NONE, ROPE_PLAIN, ROPE_LINEAR, ROPE_YARN = 0, 1, 2, 3


class RisError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(msg)
        self.status = status


class RopeCfg(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("reserved", ctypes.c_int32), ("theta", ctypes.c_double),
                ("native_len", ctypes.c_int64), ("factor", ctypes.c_double),
                ("yarn_alpha", ctypes.c_double), ("yarn_beta", ctypes.c_double)]


class MaskOpts(ctypes.Structure):
    _fields_ = [("local_window", ctypes.c_int32), ("n_anchor", ctypes.c_int32),
                ("per_head", ctypes.c_int32), ("layer_key", ctypes.c_uint32), ("sampler", ctypes.c_int32)]


class Params(ctypes.Structure):
    _fields_ = [("bmax", ctypes.c_int64), ("block", ctypes.c_int64), ("clique_pairs", ctypes.c_int64),
                ("d_clique", ctypes.c_double), ("d_global", ctypes.c_double), ("thr", ctypes.c_uint64),
                ("stream", ctypes.c_uint32), ("dense", ctypes.c_int32), ("rope_factor", ctypes.c_double),
                ("rope_mscale", ctypes.c_double), ("draws", ctypes.c_int64)]


class MaskDesc(ctypes.Structure):
    _fields_ = [("N", ctypes.c_int64), ("n_masks", ctypes.c_int32), ("heads_keyed", ctypes.c_int32),
                ("n_seeds", ctypes.c_int32), ("per_seed", ctypes.c_int32), ("col_bytes", ctypes.c_int32),
                ("dense", ctypes.c_int32), ("n_pairs", ctypes.c_int64), ("words_per_mask", ctypes.c_int64),
                ("row_ptr", ctypes.c_void_p), ("col", ctypes.c_void_p), ("bitmap", ctypes.c_void_p),
                ("params", Params), ("suffix_pairs", ctypes.c_int64)]


def rope_cfg(kind: int = ROPE_PLAIN, theta: float = 1e6, native_len: int = 32768, factor: float = 0.0,
             yarn_alpha: float = 1.0, yarn_beta: float = 32.0) -> RopeCfg:
    return RopeCfg(int(kind), 0, float(theta), int(native_len), float(factor), float(yarn_alpha),
                   float(yarn_beta))


SAMPLER_BERNOULLI, SAMPLER_DRAWS = 0, 1
PRESET_LOCAL_WINDOW, PRESET_ANCHORS = 1024, 4  # include/ris.h RIS_PRESET_*


def mask_opts(local_window: int = 1, n_anchor: int = 0, per_head: bool = False, layer_key: int = 0,
              sampler: int = SAMPLER_BERNOULLI) -> MaskOpts:
    return MaskOpts(int(local_window), int(n_anchor), int(bool(per_head)), int(layer_key), int(sampler))


def paper_geometry(per_head: bool = False, layer_key: int = 0, sampler: int = SAMPLER_BERNOULLI) -> MaskOpts:
    """The paper's local window of 1024 tokens plus global anchors over the first tokens."""
    return mask_opts(PRESET_LOCAL_WINDOW, PRESET_ANCHORS, per_head, layer_key, sampler)


_SIGS = {
    "ris_resolve_params": [ctypes.c_int64, ctypes.c_int32, ctypes.c_double, ctypes.c_void_p, ctypes.c_void_p],
    "ris_rope_freqs": [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p],
    "ris_mask_generate": [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_double, ctypes.c_void_p,
                          ctypes.c_int32, ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p],
    "ris_mask_info": [ctypes.c_void_p, ctypes.c_void_p],
    "ris_mask_free": [ctypes.c_void_p],
    "ris_rope_apply": [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                       ctypes.c_void_p, ctypes.c_void_p],
    "ris_sparse_attention_fwd": [ctypes.c_void_p] * 4 + [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                 ctypes.c_int32, ctypes.c_int32, ctypes.c_double, ctypes.c_void_p,
                                 ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p,
                                 ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p],
    "ris_attention_masked": [ctypes.c_void_p] * 5 + [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                             ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p],
    "ris_ensemble_batch": None,  # same as ris_sparse_attention_fwd
    "ris_attention_masked_noalloc": [ctypes.c_void_p] * 5 + [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                     ctypes.c_int32, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_void_p],
    "ris_noalloc_scratch_info": [ctypes.c_void_p, ctypes.c_void_p],
    "ris_shutdown": [],
    "ris_debug_fail_allocation": [ctypes.c_int64],
    "ris_debug_tile_stall": [ctypes.c_int32, ctypes.c_int64],
    "ris_kernel_timer_enable": [ctypes.c_int32],
    "ris_device_status": [ctypes.c_void_p],
    "ris_attention_design": [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int32],
    "ris_attention_masked_rows": [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64] + [ctypes.c_void_p] * 4 +
                                 [ctypes.c_int32] * 5 + [ctypes.c_void_p] * 3,
    "ris_attention_masked_local": [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int64] + [ctypes.c_void_p] * 4 +
                                  [ctypes.c_int32] * 5 + [ctypes.c_void_p] * 3,
    "ris_row_split": [ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p],
    "ris_mask_row_split": [ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p],
    "ris_kernel_timer_read": [ctypes.c_void_p, ctypes.c_void_p],
    "ris_kernel_timer_samples": [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int64],
    "ris_decode_anchor": [ctypes.c_int64, ctypes.c_int32, ctypes.c_int32, ctypes.c_double, ctypes.c_void_p,
                          ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p],
    "ris_anchor_info": [ctypes.c_void_p] * 6,
    "ris_anchor_free": [ctypes.c_void_p],
    "ris_rope_split": [ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_int64, ctypes.c_int32,
                       ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                       ctypes.c_void_p],
    "ris_decode_step": [ctypes.c_void_p] * 5 + [ctypes.c_int64, ctypes.c_int64, ctypes.c_void_p, ctypes.c_int32,
                        ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                        ctypes.c_int32, ctypes.c_int64, ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                        ctypes.c_void_p],
    "ris_probe_l2_read": [ctypes.c_int64, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p],
    "ris_probe_ffma": [ctypes.c_void_p, ctypes.c_void_p],
    "ris_probe_l2_bytes": [ctypes.c_void_p],
    "ris_memory_stats": [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32],
}


def lib():
    """Load libris.so (raises if it was not built; there is no fallback)."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(LIB_PATH):
                raise RuntimeError(f"{LIB_PATH} is missing: build it with "
                                   "`python -m paper_2607_21927_gb300.build`")
            L = ctypes.CDLL(LIB_PATH)
            for name, sig in _SIGS.items():
                fn = getattr(L, name)
                fn.argtypes = sig if sig is not None else _SIGS["ris_sparse_attention_fwd"]
                fn.restype = ctypes.c_int
            L.ris_last_error.restype = ctypes.c_char_p
            L.ris_launch_count.restype = ctypes.c_int64
            L.ris_version.restype = ctypes.c_char_p
            _lib = L
    return _lib


def ris_last_error() -> str:
    return lib().ris_last_error().decode()


def ris_launch_count() -> int:
    return int(lib().ris_launch_count())


def ris_version() -> str:
    return lib().ris_version().decode()


DESIGNS = {0: "register gather", 2: "tcgen05 masked tiles", 3: "fp32 gather",
           4: "dense suffix on tiles + register gather"}


def ris_attention_design(mask: "Mask", dtype=torch.bfloat16, head_dim: int = 128) -> int:
    """Kernel design a layer call on this mask uses (see DESIGNS)."""
    return int(lib().ris_attention_design(mask.handle, BF16 if dtype == torch.bfloat16 else F32, int(head_dim)))


def ris_device_status(stream=None) -> None:
    """Synchronise and raise RisError(RIS_ERR_DEVICE_TIMEOUT) if a device-side wait gave up."""
    _check("ris_device_status", lib().ris_device_status(_stream(stream)))


def ris_kernel_timer_enable(enable: bool = True) -> None:
    _check("ris_kernel_timer_enable", lib().ris_kernel_timer_enable(int(bool(enable))))


def ris_kernel_timer_read():
    """(summed device ms, launches) of the attention kernels recorded since the last read."""
    ms, n = ctypes.c_double(), ctypes.c_int64()
    _check("ris_kernel_timer_read", lib().ris_kernel_timer_read(ctypes.byref(ms), ctypes.byref(n)))
    return ms.value, n.value


def ris_kernel_timer_samples(capacity: int = 4096):
    """(summed device ms, launches, [ms of each recorded launch]) since the last read."""
    ms, n = ctypes.c_double(), ctypes.c_int64()
    buf = (ctypes.c_double * max(1, int(capacity)))()
    _check("ris_kernel_timer_samples", lib().ris_kernel_timer_samples(ctypes.byref(ms), ctypes.byref(n), buf,
                                                                      int(capacity)))
    return ms.value, n.value, list(buf[:min(n.value, int(capacity))])


def ris_probe_l2_read(working_set: int, pattern: int = 0, stream=None) -> float:
    """Measured read bandwidth (GB/s) over a `working_set`-byte buffer: pattern 0 streaming
    16-byte loads, 1 whole 256-byte rows at pseudo-random indices."""
    g = ctypes.c_double()
    _check("ris_probe_l2_read", lib().ris_probe_l2_read(int(working_set), int(pattern), ctypes.byref(g),
                                                        _stream(stream)))
    return g.value


def ris_probe_ffma(stream=None) -> float:
    """Measured FP32 FFMA throughput (TFLOP/s)."""
    t = ctypes.c_double()
    _check("ris_probe_ffma", lib().ris_probe_ffma(ctypes.byref(t), _stream(stream)))
    return t.value


def ris_probe_l2_bytes() -> int:
    """L2 size in bytes as the driver reports it."""
    b = ctypes.c_int64()
    _check("ris_probe_l2_bytes", lib().ris_probe_l2_bytes(ctypes.byref(b)))
    return b.value


def ris_memory_stats(reset_high_water: bool = False):
    """(bytes in use, high-water mark) of the default stream-ordered pool the library allocates from."""
    cur, high = ctypes.c_int64(), ctypes.c_int64()
    _check("ris_memory_stats", lib().ris_memory_stats(ctypes.byref(cur), ctypes.byref(high),
                                                      int(bool(reset_high_water))))
    return cur.value, high.value


def _check(name: str, st: int) -> None:
    if st != RIS_OK:
        raise RisError(st, f"{name} failed with status {st}: {ris_last_error()}")


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return BF16
    if t.dtype == torch.float32:
        return F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _seeds(seeds: Sequence[int]):
    arr = (ctypes.c_uint32 * len(seeds))(*[int(s) & 0xFFFFFFFF for s in seeds])
    return arr, len(seeds)


def _ref(x):
    return None if x is None else ctypes.byref(x)


# ----------------------------------------------------------------------------- host-side helpers
def ris_resolve_params(N: int, mode: int, density: float, rope: Optional[RopeCfg] = None) -> dict:
    p = Params()
    _check("ris_resolve_params", lib().ris_resolve_params(int(N), int(mode), float(density), _ref(rope),
                                                          ctypes.byref(p)))
    return {f: getattr(p, f) for f, _ in Params._fields_}


def ris_rope_freqs(rope: RopeCfg, N: int, head_dim: int):
    f = (ctypes.c_double * (head_dim // 2))()
    ms = ctypes.c_double()
    _check("ris_rope_freqs", lib().ris_rope_freqs(_ref(rope), int(N), int(head_dim), f, ctypes.byref(ms)))
    return list(f), ms.value


# ----------------------------------------------------------------------------- masks
class Mask:
    """A mask built by ris_mask_generate; freed by ``free()`` or when garbage collected."""

    def __init__(self, handle: ctypes.c_void_p, kv_heads: int):
        self.handle = handle
        self.kv_heads = kv_heads

    def info(self) -> MaskDesc:
        d = MaskDesc()
        _check("ris_mask_info", lib().ris_mask_info(self.handle, ctypes.byref(d)))
        return d

    def row_ptr(self) -> torch.Tensor:
        """Device row offsets as a torch view (int64, n_masks * N + 1)."""
        d = self.info()
        return _device_view(d.row_ptr, d.n_masks * d.N + 1, torch.int64)

    def cols(self) -> torch.Tensor:
        d = self.info()
        dt = torch.int16 if d.col_bytes == 2 else torch.int32
        t = _device_view(d.col, d.n_pairs, dt)
        return t.to(torch.int64) & 0xFFFF if d.col_bytes == 2 else t.to(torch.int64)

    def bitmap(self) -> torch.Tensor:
        d = self.info()
        return _device_view(d.bitmap, d.n_masks * d.words_per_mask, torch.int32)

    def free(self) -> None:
        if self.handle:
            _check("ris_mask_free", lib().ris_mask_free(self.handle))
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.free()


class _DeviceArray:
    """Exposes library-owned device memory through __cuda_array_interface__ (only ever copied)."""

    def __init__(self, ptr: int, n: int, typestr: str):
        self.__cuda_array_interface__ = {"shape": (int(n),), "typestr": typestr, "data": (int(ptr), False),
                                         "version": 3}


_TYPESTR = {torch.int64: "<i8", torch.int32: "<i4", torch.int16: "<i2"}


def _device_view(ptr: int, n: int, dtype) -> torch.Tensor:
    """A copy (owned by torch) of n elements at a library-owned device address."""
    if not ptr or n == 0:
        return torch.empty(0, dtype=dtype, device="cuda")
    torch.cuda.current_stream().synchronize()
    return torch.as_tensor(_DeviceArray(ptr, n, _TYPESTR[dtype]), device="cuda").clone()


def ris_mask_generate(N: int, kv_heads: int, mode: int, density: float, seeds: Sequence[int],
                      opts: Optional[MaskOpts] = None, per_seed: bool = False, stream=None) -> Mask:
    arr, n = _seeds(seeds)
    h = ctypes.c_void_p()
    _check("ris_mask_generate", lib().ris_mask_generate(int(N), int(kv_heads), int(mode), float(density), arr, n,
                                                        _ref(opts), int(bool(per_seed)), ctypes.byref(h),
                                                        _stream(stream)))
    return Mask(h, kv_heads)


# ----------------------------------------------------------------------------- RoPE
def ris_rope_apply(x: torch.Tensor, rope: RopeCfg, stream=None) -> torch.Tensor:
    """Rotate x [N, heads, head_dim] in place (positions 0..N-1)."""
    assert x.is_cuda and x.is_contiguous() and x.dim() == 3
    N, H, D = x.shape
    _check("ris_rope_apply", lib().ris_rope_apply(_ptr(x), _dtype(x), N, H, D, ctypes.byref(rope), _stream(stream)))
    return x


# ----------------------------------------------------------------------------- attention
def _shapes(q, k, v):
    for t in (q, k, v):
        assert t.is_cuda and t.is_contiguous() and t.dim() == 3, "q, k, v: contiguous [N, H, D] on the GPU"
    N, Hq, D = q.shape
    assert k.shape == v.shape and k.shape[0] == N and k.shape[2] == D and q.dtype == k.dtype == v.dtype
    return N, Hq, k.shape[1], D


def _alloc_out(out, shape, out_dtype, device):
    if out is None:
        out = torch.empty(shape, dtype=out_dtype, device=device)
    assert out.is_contiguous() and tuple(out.shape) == tuple(shape)
    return out


def ris_sparse_attention_fwd(q, k, v, mode: int, density: float, seeds: Sequence[int],
                             rope: Optional[RopeCfg] = None, opts: Optional[MaskOpts] = None,
                             out: Optional[torch.Tensor] = None, out_dtype=None, return_lse: bool = False,
                             stream=None):
    N, Hq, Hkv, D = _shapes(q, k, v)
    out = _alloc_out(out, (N, Hq, D), out_dtype or q.dtype, q.device)
    lse = torch.empty((Hq, N), dtype=torch.float32, device=q.device) if return_lse else None
    arr, n = _seeds(seeds)
    _check("ris_sparse_attention_fwd", lib().ris_sparse_attention_fwd(
        _ptr(q), _ptr(k), _ptr(v), _ptr(out), N, Hq, Hkv, D, int(mode), float(density), arr, n, _dtype(q),
        _dtype(out), _ref(rope), _ref(opts), _ptr(lse), _stream(stream)))
    return (out, lse) if return_lse else out


def ris_ensemble_batch(q, k, v, mode: int, density: float, seeds: Sequence[int],
                       rope: Optional[RopeCfg] = None, opts: Optional[MaskOpts] = None,
                       out: Optional[torch.Tensor] = None, out_dtype=None, return_lse: bool = False, stream=None):
    N, Hq, Hkv, D = _shapes(q, k, v)
    S = len(seeds)
    out = _alloc_out(out, (S, N, Hq, D), out_dtype or q.dtype, q.device)
    lse = torch.empty((S, Hq, N), dtype=torch.float32, device=q.device) if return_lse else None
    arr, n = _seeds(seeds)
    _check("ris_ensemble_batch", lib().ris_ensemble_batch(
        _ptr(q), _ptr(k), _ptr(v), _ptr(out), N, Hq, Hkv, D, int(mode), float(density), arr, n, _dtype(q),
        _dtype(out), _ref(rope), _ref(opts), _ptr(lse), _stream(stream)))
    return (out, lse) if return_lse else out


def ris_attention_masked(mask: Mask, q, k, v, rope: Optional[RopeCfg] = None,
                         out: Optional[torch.Tensor] = None, out_dtype=None, return_lse: bool = False,
                         stream=None):
    N, Hq, Hkv, D = _shapes(q, k, v)
    d = mask.info()
    if d.N != N:
        raise ValueError(f"q has {N} tokens, the mask was built for {d.N}")
    sets = d.n_seeds if d.per_seed else 1
    shape = (sets, N, Hq, D) if d.per_seed else (N, Hq, D)
    out = _alloc_out(out, shape, out_dtype or q.dtype, q.device)
    lse = torch.empty((sets, Hq, N) if d.per_seed else (Hq, N), dtype=torch.float32,
                      device=q.device) if return_lse else None
    _check("ris_attention_masked", lib().ris_attention_masked(
        mask.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(out), Hq, Hkv, D, _dtype(q), _dtype(out), _ref(rope),
        _ptr(lse), _stream(stream)))
    return (out, lse) if return_lse else out


def ris_attention_masked_noalloc(mask: Mask, q, k, v, out: torch.Tensor, rope: Optional[RopeCfg] = None,
                                 lse: Optional[torch.Tensor] = None, stream=None):
    """Allocation-free layer call: the caller passes every output buffer; the library's
    scratch is a fixed 64 MiB device array, and every mask runs on the gather design."""
    N, Hq, Hkv, D = _shapes(q, k, v)
    d = mask.info()
    if d.N != N:
        raise ValueError(f"q has {N} tokens, the mask was built for {d.N}")
    assert out.is_cuda and out.is_contiguous()
    _check("ris_attention_masked_noalloc", lib().ris_attention_masked_noalloc(
        mask.handle, _ptr(q), _ptr(k), _ptr(v), _ptr(out), Hq, Hkv, D, _dtype(q), _dtype(out), _ref(rope),
        _ptr(lse), _stream(stream)))
    return out


def ris_noalloc_scratch_info():
    """(device address, bytes) of the allocation-free entry point's scratch array."""
    addr, n = ctypes.c_void_p(), ctypes.c_int64()
    _check("ris_noalloc_scratch_info", lib().ris_noalloc_scratch_info(ctypes.byref(addr), ctypes.byref(n)))
    return int(addr.value or 0), int(n.value)


def ris_shutdown() -> None:
    """Release the library's cached per-device state (timer events, pool caches)."""
    _check("ris_shutdown", lib().ris_shutdown())


def ris_debug_fail_allocation(n: int) -> None:
    """Tests: the n-th stream-ordered allocation from now on fails (n < 0 disarms)."""
    _check("ris_debug_fail_allocation", lib().ris_debug_fail_allocation(int(n)))


def ris_debug_tile_stall(no_loads: bool, wait_limit_cycles: int = 0) -> None:
    """Tests: the tile kernel's loader issues no copies and its waits give up after the limit."""
    _check("ris_debug_tile_stall", lib().ris_debug_tile_stall(int(bool(no_loads)), int(wait_limit_cycles)))


# ----------------------------------------------------------------------------- Hybrid Anchor decode
class Anchor:
    """The frozen Stochastic Anchor of a generation (ris_decode_anchor); freed by ``free()``."""

    def __init__(self, handle: ctypes.c_void_p, kv_heads: int):
        self.handle = handle
        self.kv_heads = kv_heads

    def info(self):
        """(t0, heads_keyed, n_keys, keys device tensor int64, offsets device tensor int64)."""
        t0, hk, n = ctypes.c_int64(), ctypes.c_int32(), ctypes.c_int64()
        keys, off = ctypes.c_void_p(), ctypes.c_void_p()
        _check("ris_anchor_info", lib().ris_anchor_info(self.handle, ctypes.byref(t0), ctypes.byref(hk),
                                                        ctypes.byref(n), ctypes.byref(keys), ctypes.byref(off)))
        k = _device_view(keys.value, n.value, torch.int32).to(torch.int64)
        o = _device_view(off.value, hk.value + 1, torch.int64)
        return t0.value, hk.value, n.value, k, o

    def free(self) -> None:
        if self.handle:
            _check("ris_anchor_free", lib().ris_anchor_free(self.handle))
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def ris_decode_anchor(n_prefill: int, kv_heads: int, mode: int, density: float, seeds: Sequence[int],
                      opts: Optional[MaskOpts] = None, stream=None) -> Anchor:
    arr, n = _seeds(seeds)
    h = ctypes.c_void_p()
    _check("ris_decode_anchor", lib().ris_decode_anchor(int(n_prefill), int(kv_heads), int(mode), float(density),
                                                        arr, n, _ref(opts), ctypes.byref(h), _stream(stream)))
    return Anchor(h, kv_heads)


def ris_rope_split(x: torch.Tensor, n_ctx: int, rope: Optional[RopeCfg], pos0: int = 0, hi=None, lo=None,
                   split: bool = True, stream=None):
    """Rotated copy of x [n, H, D] at positions pos0.. as (hi, lo); lo (bf16 only) carries the
    residual of the bf16 rounding when split is set, else None."""
    assert x.is_cuda and x.is_contiguous() and x.dim() == 3
    n, H, D = x.shape
    hi = _alloc_out(hi, x.shape, x.dtype, x.device)
    if split and x.dtype == torch.bfloat16:
        lo = _alloc_out(lo, x.shape, torch.bfloat16, x.device)
    else:
        lo = None
    _check("ris_rope_split", lib().ris_rope_split(_ptr(x), _dtype(x), int(n), int(pos0), int(H), int(D), int(n_ctx),
                                                  _ref(rope), _ptr(hi), _ptr(lo), _stream(stream)))
    return hi, lo


def ris_decode_step(anchor: Anchor, q: torch.Tensor, k: torch.Tensor, k_lo: Optional[torch.Tensor],
                    v: torch.Tensor, t: int, window: int, n_ctx: int, rope: Optional[RopeCfg] = None,
                    out=None, out_dtype=None, return_lse: bool = False, t_dev: Optional[torch.Tensor] = None,
                    advance: bool = False, stream=None):
    """q [Hq, D] of the token at position t (not rotated); k/k_lo/v the rotated cache [T, Hkv, D].
    With t_dev (a one-element int64 CUDA tensor) the position is read on the device instead of t,
    and advance adds 1 to it once the step has run."""
    assert q.is_cuda and q.is_contiguous() and q.dim() == 2
    for x in (k, v) + ((k_lo,) if k_lo is not None else ()):
        assert x.is_cuda and x.is_contiguous() and x.dim() == 3 and x.shape == k.shape
    Hq, D = q.shape
    T, Hkv, _ = k.shape
    out = _alloc_out(out, (Hq, D), out_dtype or q.dtype, q.device)
    lse = torch.empty(Hq, dtype=torch.float32, device=q.device) if return_lse else None
    if t_dev is not None:
        assert t_dev.is_cuda and t_dev.dtype == torch.int64 and t_dev.numel() == 1
    _check("ris_decode_step", lib().ris_decode_step(
        anchor.handle, _ptr(q), _ptr(k), _ptr(k_lo), _ptr(v), int(T), int(t), _ptr(t_dev), int(bool(advance)),
        int(window), int(Hq), int(Hkv), int(D), _dtype(q), _dtype(out), int(n_ctx), _ref(rope), _ptr(out), _ptr(lse),
        _stream(stream)))
    return (out, lse) if return_lse else out


# ----------------------------------------------------------------------------- row ranges
def ris_attention_masked_rows(mask: Mask, row_begin: int, row_end: int, q, k, v, out: torch.Tensor,
                              rope: Optional[RopeCfg] = None, lse: Optional[torch.Tensor] = None, stream=None):
    """Rows row_begin .. row_end-1 of ris_attention_masked into `out` (other rows untouched)."""
    N, Hq, Hkv, D = _shapes(q, k, v)
    assert out.is_cuda and out.is_contiguous()
    _check("ris_attention_masked_rows", lib().ris_attention_masked_rows(
        mask.handle, int(row_begin), int(row_end), _ptr(q), _ptr(k), _ptr(v), _ptr(out), Hq, Hkv, D, _dtype(q),
        _dtype(out), _ref(rope), _ptr(lse), _stream(stream)))
    return out


def ris_attention_masked_local(mask: Mask, row_begin: int, row_end: int, q_rows, k, v, out_rows=None,
                               rope: Optional[RopeCfg] = None, out_dtype=None, return_lse: bool = False, stream=None):
    """Rows row_begin .. row_end-1 with only those rows of q in memory (q_rows [rows, Hq, D]);
    k and v hold every position. Returns out_rows [rows, Hq, D] (and lse [Hq, rows])."""
    for t in (q_rows, k, v):
        assert t.is_cuda and t.is_contiguous() and t.dim() == 3
    rows, Hq, D = q_rows.shape
    Hkv = k.shape[1]
    assert rows == row_end - row_begin and k.shape == v.shape and k.shape[2] == D
    out_rows = _alloc_out(out_rows, (rows, Hq, D), out_dtype or q_rows.dtype, q_rows.device)
    lse = torch.empty((Hq, rows), dtype=torch.float32, device=q_rows.device) if return_lse else None
    _check("ris_attention_masked_local", lib().ris_attention_masked_local(
        mask.handle, int(row_begin), int(row_end), _ptr(q_rows), _ptr(k), _ptr(v), _ptr(out_rows), Hq, Hkv, D,
        _dtype(q_rows), _dtype(out_rows), _ref(rope), _ptr(lse), _stream(stream)))
    return (out_rows, lse) if return_lse else out_rows


def ris_row_split(row_ptr, parts: int):
    """Balanced row bounds (parts + 1 of them) from a host row_ptr of N + 1 offsets."""
    import numpy as np

    rp = np.ascontiguousarray(np.asarray(row_ptr, dtype=np.int64))
    b = np.empty(int(parts) + 1, dtype=np.int64)
    _check("ris_row_split", lib().ris_row_split(rp.ctypes.data, int(rp.shape[0] - 1), int(parts), b.ctypes.data))
    return b.tolist()


def ris_mask_row_split(mask: Mask, parts: int):
    """Balanced row bounds (parts + 1 of them) by the mask's sampled-pair counts."""
    b = (ctypes.c_int64 * (int(parts) + 1))()
    _check("ris_mask_row_split", lib().ris_mask_row_split(mask.handle, int(parts), b))
    return list(b)

