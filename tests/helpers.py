"""Shared test helpers: seeded inputs, oracle adapters and the tolerances of the parity bar."""
import numpy as np
import torch

import oracle as ora
from paper_2607_21927_gb300 import inputs

# Tolerances against the fp64 oracle.
#   bf16 inputs, fp32 accumulation: max-abs <= 1e-2 and relative L2 <= 5e-3;
#   fp32 inputs: relative L2 <= 1e-5.
# A bf16 OUTPUT adds its own rounding: half an ulp, 2^-9 |o| (relative), which for |o| > 2.56
# alone exceeds 1e-2; with a bf16 output the max-abs bar becomes 1e-2 + 2^-8 |o_ref| (half an
# ulp of the output plus the same budget again for the fp32 value it was rounded from).
BF16_MAX_ABS = 1e-2
BF16_REL_L2 = 5e-3
F32_REL_L2 = 1e-5


def rel_l2(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.linalg.norm((got - ref).ravel()) / max(np.linalg.norm(ref.ravel()), 1e-300))


def check_bf16_path(got, ref, out_bf16=False):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    err = np.abs(got - ref)
    bound = BF16_MAX_ABS + (2.0 ** -8) * np.abs(ref) if out_bf16 else BF16_MAX_ABS
    bad = err > bound
    assert not bad.any(), (f"max-abs {err.max():.3e} over bound at {int(bad.sum())} elements "
                           f"(worst ref {ref.ravel()[np.argmax((err - bound).ravel())]:.3f})")
    r = rel_l2(got, ref)
    assert r <= BF16_REL_L2, f"relative L2 {r:.3e} > {BF16_REL_L2}"
    return float(err.max()), r


def check_f32_path(got, ref):
    r = rel_l2(got, ref)
    assert r <= F32_REL_L2, f"relative L2 {r:.3e} > {F32_REL_L2}"
    return r


def to_np(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


def make_inputs(N, Hq, Hkv, D, dtype=torch.bfloat16, seed=0, outliers=False, device="cuda"):
    """Seeded q, k, v on the GPU plus their exact fp64 host copies for the oracle."""
    gen_dev = "cuda" if (device == "cuda" and N * (Hq + 2 * Hkv) * D > (1 << 24)) else "cpu"
    q, k, v = inputs.make_qkv(N, Hq, Hkv, D, dtype=dtype, seed=seed, outliers=outliers, device=gen_dev)
    qd, kd, vd = (t.to(device).contiguous() for t in (q, k, v))
    return (qd, kd, vd), (to_np(q), to_np(k), to_np(v))


def oracle_rope(kind, theta, native_len, factor=0.0):
    if kind == 0:
        return None
    return ora.RopeCfg(kind=kind, theta=theta, native_len=native_len, factor=factor)


def row_word_offset(i):
    a, b = i >> 5, i & 31
    return i + 16 * a * (a - 1) + a * b


def sample_rows(N, n, seed=0):
    """First, last, a few small and n random rows (sorted, unique)."""
    rng = np.random.default_rng(seed)
    base = [0, 1, 2, 31, 32, 33, N // 2, N - 2, N - 1]
    rows = np.unique(np.clip(np.concatenate([base, rng.integers(0, N, size=n)]), 0, N - 1))
    return rows.astype(np.int64)
