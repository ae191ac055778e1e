"""fp64 CPU oracle for RIS prefill sparse attention.

TEST INFRASTRUCTURE. Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` import this package. The product path (the CUDA library under
``paper_2607_21927_gb300``) never imports it; the two share no code.

The arithmetic lives in ``ris_oracle.c`` (plain C, fp64, OpenMP over rows). This module
only marshals numpy arrays and composes the steps in the order the paper gives them:
draw each seed's pairs, OR them into one master mask (Methods, "Memory-Bounded
Geometry Generation"), rotate q and k (Methods, "Dynamic RoPE Scaling"), then one
softmax over each row's whole key set (Methods, "Pre-Fusion Unified Softmax").
"""
from __future__ import annotations

import ctypes
import math
import os
import subprocess
import threading
from dataclasses import dataclass, field
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ris_oracle.c")
_LIB = os.path.join(_HERE, "libris_oracle.so")
_lock = threading.Lock()
_lib = None

MODE_STOCHASTIC, MODE_STRUCTURAL, MODE_DENSE = 0, 1, 2
ROPE_NONE, ROPE_PLAIN, ROPE_LINEAR, ROPE_YARN = 0, 1, 2, 3


def build(force: bool = False) -> str:
    """Compile ris_oracle.c into libris_oracle.so beside it (gcc, fp64, OpenMP)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        subprocess.check_call(
            ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
        )
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i64, i32, f64 = ctypes.c_int64, ctypes.c_int32, ctypes.c_double
            lib.ora_philox_batch.argtypes = [i64, P, P, P]
            lib.ora_threshold.argtypes = [f64]
            lib.ora_threshold.restype = ctypes.c_uint64
            lib.ora_structural.argtypes = [i64, f64, P, P, P, P, P]
            lib.ora_mask_counts.argtypes = [P, P, i64, P]
            lib.ora_mask_cols.argtypes = [P, P, i64, P, P]
            lib.ora_mask_bits.argtypes = [P, P, i64, i64, P]
            lib.ora_rope_freqs.argtypes = [i32, f64, i64, f64, f64, f64, i32, P, P]
            lib.ora_rope_apply.argtypes = [P, P, i64, i32, i32, P, f64]
            lib.ora_attention.argtypes = [P, P, P, i64, i32, i32, i32, i64, P, P, P, P]
            lib.ora_set_threads.argtypes = [i32]
            lib.ora_get_threads.restype = i32
            _lib = lib
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def set_threads(n: int) -> None:
    _load().ora_set_threads(int(n))


def get_threads() -> int:
    return int(_load().ora_get_threads())


# ----------------------------------------------------------------------------- Philox
def philox(ctr: np.ndarray, key: np.ndarray) -> np.ndarray:
    """Philox4x32-10 of each row: ctr uint32[n,4], key uint32[n,2] -> uint32[n,4]."""
    ctr = np.ascontiguousarray(ctr, dtype=np.uint32).reshape(-1, 4)
    key = np.ascontiguousarray(key, dtype=np.uint32).reshape(-1, 2)
    assert ctr.shape[0] == key.shape[0]
    out = np.empty_like(ctr)
    _load().ora_philox_batch(ctr.shape[0], _p(ctr), _p(key), _p(out))
    return out


def threshold(p: float) -> int:
    """Keep-threshold on a uniform 32-bit word for probability p."""
    return int(_load().ora_threshold(float(p)))


def structural(N: int, d: float) -> dict:
    """Structural-mode geometry: B_max = K, block size B, clique pairs C, d_clique, d_global."""
    vals = [ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64(), ctypes.c_double(), ctypes.c_double()]
    _load().ora_structural(int(N), float(d), *[ctypes.byref(v) for v in vals])
    K, B, C, dc, dg = [v.value for v in vals]
    return {"K": K, "B": B, "C": C, "d_clique": dc, "d_global": dg}


def union_coverage(d: float, n_seeds: int) -> float:
    """Expected union coverage U = 1 - (1 - d)^n_seeds (Eq. union_coverage)."""
    return 1.0 - (1.0 - d) ** n_seeds


# ----------------------------------------------------------------------------- masks
class _Spec(ctypes.Structure):
    _fields_ = [
        ("N", ctypes.c_int64),
        ("mode", ctypes.c_int32),
        ("n_seeds", ctypes.c_int32),
        ("density", ctypes.c_double),
        ("seeds", ctypes.c_void_p),
        ("seed_index", ctypes.c_int32),
        ("local_window", ctypes.c_int32),
        ("n_anchor", ctypes.c_int32),
        ("head_key", ctypes.c_uint32),
        ("layer_key", ctypes.c_uint32),
        ("sampler", ctypes.c_int32),
    ]


@dataclass
class MaskSpec:
    """One RIS mask: mode, density d, the ensemble seeds and the forced set."""

    N: int
    mode: int
    density: float
    seeds: Sequence[int]
    seed_index: int = -1  # -1: union of all seeds (master mask); s: seed s alone
    local_window: int = 1
    n_anchor: int = 0
    head_key: int = 0
    layer_key: int = 0
    sampler: int = 0  # 0: Bernoulli test per causal pair; 1: index draws with replacement
    _seeds_arr: np.ndarray = field(default=None, repr=False)

    def _c(self) -> _Spec:
        self._seeds_arr = np.ascontiguousarray(np.asarray(self.seeds, dtype=np.uint32))
        return _Spec(
            int(self.N), int(self.mode), len(self.seeds), float(self.density),
            self._seeds_arr.ctypes.data, int(self.seed_index), int(self.local_window),
            int(self.n_anchor), int(self.head_key), int(self.layer_key), int(self.sampler),
        )


def _rows(spec: MaskSpec, rows) -> np.ndarray:
    if rows is None:
        rows = np.arange(spec.N, dtype=np.int64)
    return np.ascontiguousarray(np.asarray(rows, dtype=np.int64))


def mask_counts(spec: MaskSpec, rows=None) -> np.ndarray:
    rows = _rows(spec, rows)
    out = np.empty(rows.shape[0], dtype=np.int64)
    cs = spec._c()
    _load().ora_mask_counts(ctypes.byref(cs), _p(rows), rows.shape[0], _p(out))
    return out


def mask_cols(spec: MaskSpec, rows=None):
    """Key lists of the given rows: (off int64[nrows+1], cols int64[off[-1]]), ascending."""
    rows = _rows(spec, rows)
    counts = mask_counts(spec, rows)
    off = np.zeros(rows.shape[0] + 1, dtype=np.int64)
    np.cumsum(counts, out=off[1:])
    cols = np.empty(int(off[-1]), dtype=np.int64)
    cs = spec._c()
    _load().ora_mask_cols(ctypes.byref(cs), _p(rows), rows.shape[0], _p(off), _p(cols))
    return off, cols


def mask_bits(spec: MaskSpec, rows=None, words_per_row: Optional[int] = None) -> np.ndarray:
    """Bitmap words uint32[nrows, words_per_row]; bit j%32 of word j//32 is pair (i, j)."""
    rows = _rows(spec, rows)
    if words_per_row is None:
        words_per_row = (spec.N + 31) // 32
    out = np.empty((rows.shape[0], words_per_row), dtype=np.uint32)
    cs = spec._c()
    _load().ora_mask_bits(ctypes.byref(cs), _p(rows), rows.shape[0], int(words_per_row), _p(out))
    return out


def mask_dense(spec: MaskSpec) -> np.ndarray:
    """The whole mask as bool[N, N] (small N only)."""
    off, cols = mask_cols(spec)
    m = np.zeros((spec.N, spec.N), dtype=bool)
    rows = np.repeat(np.arange(spec.N), np.diff(off))
    m[rows, cols] = True
    return m


# ----------------------------------------------------------------------------- RoPE
@dataclass
class RopeCfg:
    kind: int = ROPE_PLAIN
    theta: float = 1e6
    native_len: int = 32768
    factor: float = 0.0  # <= 0: resolved as max(1, N / native_len)
    alpha: float = 1.0
    beta: float = 32.0


def resolve_factor(cfg: RopeCfg, N: int) -> float:
    """Extension factor: requested window over the native limit (Methods, Dynamic RoPE Scaling)."""
    if cfg.factor > 0:
        return float(cfg.factor)
    return max(1.0, float(N) / float(cfg.native_len))


def rope_freqs(cfg: RopeCfg, N: int, D: int):
    s = resolve_factor(cfg, N)
    f = np.empty(D // 2, dtype=np.float64)
    ms = ctypes.c_double()
    _load().ora_rope_freqs(int(cfg.kind), float(cfg.theta), int(cfg.native_len), s,
                           float(cfg.alpha), float(cfg.beta), int(D), _p(f), ctypes.byref(ms))
    return f, ms.value


def rope(x: np.ndarray, pos, cfg: Optional[RopeCfg], N: int) -> np.ndarray:
    """Rotated fp64 copy of x[n, H, D] at positions pos[n]; cfg None or kind 0 is the identity."""
    x = np.array(x, dtype=np.float64, order="C", copy=True)
    if cfg is None or cfg.kind == ROPE_NONE:
        return x
    n, H, D = x.shape
    f, ms = rope_freqs(cfg, N, D)
    pos = np.ascontiguousarray(np.asarray(pos, dtype=np.float64))
    assert pos.shape[0] == n
    _load().ora_rope_apply(_p(x), _p(pos), n, H, D, _p(f), ms)
    return x


# ----------------------------------------------------------------------------- attention
def attention(q_rows: np.ndarray, k: np.ndarray, v: np.ndarray, off: np.ndarray, cols: np.ndarray):
    """Masked softmax attention of already-rotated rows: returns (out[nrows,Hq,D], lse[nrows,Hq])."""
    q_rows = np.ascontiguousarray(q_rows, dtype=np.float64)
    k = np.ascontiguousarray(k, dtype=np.float64)
    v = np.ascontiguousarray(v, dtype=np.float64)
    off = np.ascontiguousarray(off, dtype=np.int64)
    cols = np.ascontiguousarray(cols, dtype=np.int64)
    nrows, Hq, D = q_rows.shape
    N, Hkv, Dk = k.shape
    assert Dk == D and v.shape == k.shape and off.shape[0] == nrows + 1
    out = np.empty((nrows, Hq, D), dtype=np.float64)
    lse = np.empty((nrows, Hq), dtype=np.float64)
    _load().ora_attention(_p(q_rows), _p(k), _p(v), N, Hq, Hkv, D, nrows, _p(off), _p(cols),
                          _p(out), _p(lse))
    return out, lse


def sparse_attention(q, k, v, spec: MaskSpec, rope_cfg: Optional[RopeCfg] = None, rows=None):
    """Whole path for the given rows: mask rows, RoPE of q rows and all of k, PFUS attention.

    q: [N, Hq, D], k, v: [N, Hkv, D] (any float dtype; values are taken exactly in fp64).
    Returns (out[nrows, Hq, D], lse[nrows, Hq], off, cols).
    """
    N = spec.N
    rows = _rows(spec, rows)
    q = np.asarray(q)
    k = np.asarray(k)
    qr = rope(q[rows], rows.astype(np.float64), rope_cfg, N)
    kr = rope(k, np.arange(N, dtype=np.float64), rope_cfg, N)
    off, cols = mask_cols(spec, rows)
    out, lse = attention(qr, kr, np.asarray(v, dtype=np.float64), off, cols)
    return out, lse, off, cols



# ----------------------------------------------------------------------------- Hybrid Anchor decode
def decode_anchor(spec: MaskSpec) -> np.ndarray:
    """Stochastic Anchor (Methods, "Hybrid Anchor and Pre-Fusion Unified Softmax"): the key set
    of the first generated token, at position t0 = spec.N (the prefill length), frozen for the
    rest of the generation. Reading: it is row t0 of the RIS mask with the prefill's parameters
    (mode, density, seeds, anchors, keys, sampler) and without its local window, i.e. every
    kept key j < t0; the local part is the decode step's own sliding window."""
    t0 = int(spec.N)
    s = MaskSpec(N=spec.N, mode=spec.mode, density=spec.density, seeds=spec.seeds, seed_index=spec.seed_index,
                 local_window=1, n_anchor=spec.n_anchor, head_key=spec.head_key, layer_key=spec.layer_key,
                 sampler=spec.sampler)
    off, cols = mask_cols(s, np.array([t0], dtype=np.int64))
    return cols[cols < t0]


def decode_keys(anchor: np.ndarray, t: int, window: int) -> np.ndarray:
    """Keys of the token at position t: the frozen anchor merged with the Dynamic Local Window
    {t - window < j <= t}, duplicates removed, ascending (the paper's unique() merge)."""
    win = np.arange(max(0, t - window + 1), t + 1, dtype=np.int64)
    return np.union1d(np.asarray(anchor, dtype=np.int64), win)


def decode_step(q_t, k, v, t: int, anchor: np.ndarray, window: int, rope_cfg: Optional[RopeCfg], n_ctx: int):
    """One generated token: q_t [Hq, D] at position t attends, with one softmax (PFUS), to the
    merged key set over the cache k, v [T, Hkv, D] (T > t). RoPE of q at position t and of the
    cache at positions 0..T-1, with the extension factor resolved for n_ctx tokens.
    Returns (out[Hq, D], lse[Hq], keys)."""
    k = np.asarray(k)
    T = k.shape[0]
    assert t < T
    keys = decode_keys(anchor, t, window)
    qr = rope(np.asarray(q_t)[None], np.array([float(t)]), rope_cfg, n_ctx)
    kr = rope(k, np.arange(T, dtype=np.float64), rope_cfg, n_ctx)
    out, lse = attention(qr, kr, np.asarray(v, dtype=np.float64), np.array([0, keys.shape[0]]), keys)
    return out[0], lse[0], keys
