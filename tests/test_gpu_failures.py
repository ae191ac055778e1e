"""Failure detection without a GPU fault.

- Host side: every entry point that allocates must turn a failed stream-ordered allocation
  into RIS_ERR_OOM, leave its output handle NULL and release on its stream what it had
  already taken. The failure is injected on the host (ris_debug_fail_allocation): the n-th
  allocation from now fails, for every n until the call needs fewer allocations than n.
- Device side: the tile kernel's mbarrier waits are bounded. With its loader switched off
  (ris_debug_tile_stall), the first wait on a copy that was never issued gives up after a
  few thousand cycles: the kernel sets its error word, releases its tensor memory and
  returns, ris_device_status reports RIS_ERR_DEVICE_TIMEOUT, and the context stays usable
  (the next launches allocate tensor memory again and match the oracle).
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as ora
from helpers import check_bf16_path, make_inputs, oracle_rope, to_np
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def _in_use():
    torch.cuda.synchronize()
    return ris.ris_memory_stats()[0]


def _sweep(call, max_allocs=64):
    """Fail allocation n = 0, 1, ... of `call` until it succeeds; return (failures, result)."""
    base = _in_use()
    n = 0
    try:
        while True:
            ris.ris_debug_fail_allocation(n)
            try:
                res = call()
            except ris.RisError as e:
                assert e.status == ris.RIS_ERR_OOM, f"allocation {n}: status {e.status} ({e})"
                assert _in_use() == base, f"allocation {n}: pool memory leaked"
                n += 1
                assert n < max_allocs
                continue
            return n, res
    finally:
        ris.ris_debug_fail_allocation(-1)


def test_mask_generate_oom_leaves_null_and_frees():
    L = ris.lib()
    for N, mode, sampler in ((3000, 0, 0), (3000, 1, 1)):
        seeds = (ctypes.c_uint32 * 3)(1, 2, 3)
        opts = ris.mask_opts(sampler=sampler)

        def call():
            h = ctypes.c_void_p(12345)
            st = L.ris_mask_generate(N, 2, mode, 0.05, seeds, 3, ctypes.byref(opts), 0, ctypes.byref(h),
                                     ris._stream(None))
            if st != ris.RIS_OK:
                assert h.value is None, "out_mask not NULL after a failure"
                raise ris.RisError(st, ris.ris_last_error())
            return h
        fails, h = _sweep(call)
        assert fails >= 3  # bitmap, row counts, scan partials, key lists
        assert L.ris_mask_free(h) == ris.RIS_OK


def test_attention_calls_oom():
    N, Hq, Hkv, D = 1500, 6, 2, 128
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=3, outliers=True)
    rope = ris.rope_cfg(3, 1e6, 256)
    # each call allocates a mask and / or rotated q~ / k~ (and the split's partial outputs)
    fails, out = _sweep(lambda: ris.ris_sparse_attention_fwd(q, k, v, 0, 0.02, [1, 2], rope=rope))
    assert fails >= 5
    fails, out2 = _sweep(lambda: ris.ris_ensemble_batch(q, k, v, 0, 0.02, [1, 2], rope=rope))
    assert fails >= 5
    for mode, d, S in ((0, 0.02, 2), (1, 0.1, 1), (0, 0.5, 2)):  # gather, dense-suffix split, tiles
        m = ris.ris_mask_generate(N, Hkv, mode, d, list(range(S)))
        fails, _ = _sweep(lambda: ris.ris_attention_masked(m, q, k, v, rope=rope))
        assert fails >= 3
        o = torch.zeros(N, Hq, D, dtype=torch.bfloat16, device="cuda")
        fails, _ = _sweep(lambda: ris.ris_attention_masked_rows(m, 100, 900, q, k, v, o, rope=rope))
        assert fails >= 3
        m.free()
    torch.cuda.synchronize()


def test_decode_calls_oom():
    L = ris.lib()
    T, Hq, Hkv, D, t0 = 1200, 6, 2, 128, 1000
    seeds = (ctypes.c_uint32 * 2)(5, 6)

    def anchor():
        h = ctypes.c_void_p(777)
        st = L.ris_decode_anchor(t0, Hkv, 0, 0.05, seeds, 2, None, ctypes.byref(h), ris._stream(None))
        if st != ris.RIS_OK:
            assert h.value is None, "anchor not NULL after a failure"
            raise ris.RisError(st, ris.ris_last_error())
        return ris.Anchor(h, Hkv)
    fails, an = _sweep(anchor)
    assert fails >= 3
    (q, k, v), _ = make_inputs(T, Hq, Hkv, D, seed=8)
    rope = ris.rope_cfg(3, 1e6, 512)
    kh, kl = ris.ris_rope_split(k, T, rope)
    qt = q[t0 + 5].contiguous()
    fails, out = _sweep(lambda: ris.ris_decode_step(an, qt, kh, kl, v, t0 + 5, 64, T, rope=rope))
    assert fails == 1  # the partials buffer of the first step
    an.free()


def test_tile_wait_gives_up_and_context_survives():
    N, Hq, Hkv, D = 600, 12, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=23, outliers=True)
    rope = ris.rope_cfg(3, 1e6, 256)
    m = ris.ris_mask_generate(N, Hkv, 0, 0.5, [1, 2])
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 2  # the tile kernel
    ris.ris_device_status()
    try:
        ris.ris_debug_tile_stall(True, 4000)
        ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
        torch.cuda.synchronize()
    finally:
        ris.ris_debug_tile_stall(False, 0)
    with pytest.raises(ris.RisError) as e:
        ris.ris_device_status()
    assert e.value.status == ris.RIS_ERR_DEVICE_TIMEOUT
    ris.ris_device_status()  # the word was cleared by the read
    # tensor memory was released: the tile kernel runs again and is correct
    for _ in range(2):
        out = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
        torch.cuda.synchronize()
        ris.ris_device_status()
    spec = ora.MaskSpec(N=N, mode=0, density=0.5, seeds=[1, 2])
    ref, _, _, _ = ora.sparse_attention(qn, kn, vn, spec, oracle_rope(3, 1e6, 256))
    check_bf16_path(to_np(out), ref)
    m.free()


def test_shutdown_releases_caches_and_library_stays_usable():
    N, Hq, Hkv, D = 900, 6, 2, 128
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=5, outliers=True)
    a = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.05, [1], out_dtype=torch.float32)
    before = _in_use()
    ris.ris_kernel_timer_enable(True)
    ris.ris_sparse_attention_fwd(q, k, v, 0, 0.05, [1], out_dtype=torch.float32)
    torch.cuda.synchronize()
    ris.ris_shutdown()
    assert ris.ris_kernel_timer_read() == (0.0, 0)  # the timer was switched off and cleared
    b = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.05, [1], out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(a, b)
    assert _in_use() == before  # shutdown frees no live object and the calls leave nothing behind
