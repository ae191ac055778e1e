"""The C ABI without a GPU: the library loads, exports every declared symbol, validates its
arguments before any launch, and its host-side parameter resolution agrees with the oracle."""
import ctypes
import math
import os
import re

import numpy as np
import pytest

import oracle as ora
from conftest import ROOT, golden


@pytest.fixture(scope="module")
def ris():
    from paper_2607_21927_gb300 import build, ris as binding

    build.build()
    return binding


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "ris.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ris_[a-z0-9_]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(ris):
    names = declared_symbols()
    assert len(names) >= 12
    L = ris.lib()
    for n in names:
        assert hasattr(L, n), n


def test_invalid_arguments_launch_nothing(ris):
    L = ris.lib()
    before = ris.ris_launch_count()
    buf = (ctypes.c_uint8 * 256)()
    p = ctypes.addressof(buf)
    p16 = p + (-p % 16)
    seeds = (ctypes.c_uint32 * 2)(1, 2)
    args = dict(q=p16, k=p16, v=p16, out=p16, N=64, heads=4, kv_heads=2, D=128, mode=0, d=0.05, seeds=seeds,
                S=2, dt=1, odt=0)

    def call(**kw):
        a = dict(args, **kw)
        return L.ris_sparse_attention_fwd(a["q"], a["k"], a["v"], a["out"], a["N"], a["heads"], a["kv_heads"],
                                          a["D"], a["mode"], a["d"], a["seeds"], a["S"], a["dt"], a["odt"],
                                          None, None, None, None)

    cases = [dict(q=None), dict(out=p16 + 4), dict(N=0), dict(heads=5), dict(D=96), dict(mode=3), dict(d=0.0),
             dict(d=1.5), dict(d=float("nan")), dict(S=0), dict(S=257), dict(seeds=None), dict(dt=2),
             dict(odt=7)]
    for c in cases:
        assert call(**c) == ris.RIS_ERR_INVALID, (c, ris.ris_last_error())
        assert ris.ris_last_error() != ""
    # more than 8 query heads per KV head: bf16 only (the tile design)
    assert call(heads=32, kv_heads=2, dt=0) == ris.RIS_ERR_UNSUPPORTED
    bad_rope = ris.rope_cfg(3, 1e6, 32768)
    bad_rope.yarn_beta = 0.5
    st = L.ris_sparse_attention_fwd(p16, p16, p16, p16, 64, 4, 2, 128, 0, 0.05, seeds, 2, 1, 0,
                                    ctypes.byref(bad_rope), None, None, None)
    assert st == ris.RIS_ERR_INVALID
    bad_opts = ris.mask_opts(local_window=0)
    h = ctypes.c_void_p()
    assert L.ris_mask_generate(64, 1, 0, 0.1, seeds, 2, ctypes.byref(bad_opts), 0, ctypes.byref(h), None) \
        == ris.RIS_ERR_INVALID
    assert h.value is None
    bad_sampler = ris.mask_opts(sampler=2)
    assert L.ris_mask_generate(64, 1, 0, 0.1, seeds, 2, ctypes.byref(bad_sampler), 0, ctypes.byref(h), None) \
        == ris.RIS_ERR_INVALID
    assert h.value is None
    assert L.ris_rope_apply(None, 1, 10, 1, 128, ctypes.byref(ris.rope_cfg()), None) == ris.RIS_ERR_INVALID
    assert ris.ris_launch_count() == before


def test_compute_without_device_fails_loudly(ris):
    """No CPU fallback: on a host without a GPU a valid call reports a CUDA error."""
    import torch

    if torch.cuda.is_available():
        pytest.skip("host has a GPU")
    seeds = (ctypes.c_uint32 * 1)(1)
    h = ctypes.c_void_p()
    st = ris.lib().ris_mask_generate(1000, 1, 0, 0.1, seeds, 1, None, 0, ctypes.byref(h), None)
    assert st == ris.RIS_ERR_CUDA and h.value is None


@pytest.mark.parametrize("N", [17, 1000, 16384, 65536, 100003])
@pytest.mark.parametrize("d", [0.001, 0.01, 0.05, 0.37])
def test_resolve_params_agrees_with_oracle(ris, N, d):
    p = ris.ris_resolve_params(N, 1, d)
    g = ora.structural(N, d)
    assert (p["bmax"], p["block"], p["clique_pairs"]) == (g["K"], g["B"], g["C"])
    assert p["d_clique"] == g["d_clique"] and p["d_global"] == g["d_global"]
    assert p["thr"] == ora.threshold(g["d_global"]) and p["stream"] == 1
    # index-draw sampler: K draws per row, the oracle's count for the Structural global part
    assert p["draws"] == math.floor(g["d_global"] * N + 0.5)
    assert ris.ris_resolve_params(N, 0, d)["draws"] == math.floor(d * N + 0.5)
    s = ris.ris_resolve_params(N, 0, d)
    assert s["thr"] == ora.threshold(d) and s["stream"] == 0 and s["dense"] == 0
    assert ris.ris_resolve_params(N, 0, 1.0)["dense"] == 1
    assert ris.ris_resolve_params(N, 2, 0.01)["dense"] == 1


def test_resolve_params_bmax_table(ris):
    for N, dpct, bmax in golden("bmax_table.txt"):
        assert ris.ris_resolve_params(int(N), 1, float(dpct) / 100)["block"] == int(bmax)


@pytest.mark.parametrize("kind,N,native", [(1, 1000, 4096), (2, 65536, 32768), (3, 65536, 32768), (3, 16384, 2048),
                                           (3, 100, 2048)])
def test_rope_freqs_agree_with_oracle(ris, kind, N, native):
    for D, theta in ((128, 1e6), (64, 1e4)):
        f, ms = ris.ris_rope_freqs(ris.rope_cfg(kind, theta, native), N, D)
        fo, mso = ora.rope_freqs(ora.RopeCfg(kind=kind, theta=theta, native_len=native), N, D)
        np.testing.assert_allclose(f, fo, rtol=1e-15)
        assert ms == pytest.approx(mso, rel=1e-15)


def test_explicit_factor_overrides_auto(ris):
    p = ris.ris_resolve_params(1000, 0, 0.1, ris.rope_cfg(2, 1e4, 100, factor=3.0))
    assert p["rope_factor"] == 3.0
    p = ris.ris_resolve_params(1000, 0, 0.1, ris.rope_cfg(3, 1e4, 100))
    assert p["rope_factor"] == 10.0 and p["rope_mscale"] == pytest.approx(0.1 * math.log(10) + 1)
