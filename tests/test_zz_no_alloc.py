"""The allocation-free layer entry point, ris_attention_masked_noalloc, through the C ABI.

It serves callers that may not allocate device memory while a layer runs (an inference
engine's enqueue callback, a server with a memory plan fixed at load time). Its outputs and
log-sum-exp must match the fp64 oracle within the parity tolerance, and its outputs must match
ris_attention_masked's, on consecutive calls that reuse the same fixed scratch array; sizes
beyond that array must be refused before any launch. Every mask, dense ones included, runs on
the gather design here. This file is collected last so that a failure here never hides the
other GPU tests.
"""
import numpy as np
import pytest
import torch

import oracle as ora
from helpers import (BF16_MAX_ABS, BF16_REL_L2, F32_REL_L2, check_bf16_path, check_f32_path, make_inputs,
                     oracle_rope, rel_l2, to_np)
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def _compare(got, ref, fp32):
    g, r = to_np(got), to_np(ref)
    if fp32:
        assert rel_l2(g, r) <= F32_REL_L2
    else:
        assert np.abs(g - r).max() <= BF16_MAX_ABS and rel_l2(g, r) <= BF16_REL_L2


@pytest.mark.parametrize("dtype,Hq,Hkv,D,mode", [(torch.bfloat16, 12, 2, 128, 0), (torch.float32, 4, 1, 64, 1)])
def test_noalloc_matches_pool_path_and_oracle_on_consecutive_calls(dtype, Hq, Hkv, D, mode):
    N = 3000
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 1024)
    seeds = [0, 1, 2]
    mask = ris.ris_mask_generate(N, Hkv, mode, 0.03, seeds)
    fp32 = dtype == torch.float32
    addr0, nbytes = ris.ris_noalloc_scratch_info()
    assert addr0 != 0 and nbytes == 64 << 20
    for call, seed in enumerate((11, 12)):  # two calls in a row, different inputs
        (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, dtype=dtype, seed=seed, outliers=not fp32)
        ref = ris.ris_attention_masked(mask, q, k, v, rope=rope, out_dtype=torch.float32)
        out = torch.full((N, Hq, D), float("nan"), dtype=torch.float32, device="cuda")
        lse = torch.full((Hq, N), float("nan"), dtype=torch.float32, device="cuda")
        ris.ris_attention_masked_noalloc(mask, q, k, v, out, rope=rope, lse=lse)
        torch.cuda.synchronize()
        assert torch.isfinite(out).all() and torch.isfinite(lse).all(), f"call {call}"
        _compare(out, ref, fp32)
        spec = ora.MaskSpec(N=N, mode=mode, density=0.03, seeds=seeds)
        o_ref, lse_ref, _, _ = ora.sparse_attention(qn, kn, vn, spec, oracle_rope(3, 1e6, 1024))
        if fp32:
            check_f32_path(to_np(out), o_ref)
            np.testing.assert_allclose(to_np(lse).T, lse_ref, rtol=1e-5, atol=1e-5)
        else:
            check_bf16_path(to_np(out), o_ref)
            np.testing.assert_allclose(to_np(lse).T, lse_ref, rtol=0, atol=2e-3)
    assert ris.ris_noalloc_scratch_info()[0] == addr0  # same context: the same array
    mask.free()


def test_noalloc_dense_mask_against_oracle():
    """A dense mask (density 1) runs the gather's dense branch here (ris_attention_masked takes
    the tiles): outputs and log-sum-exp against the oracle, bf16 output."""
    N, Hq, Hkv, D = 700, 12, 2, 128
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 256)
    mask = ris.ris_mask_generate(N, Hkv, ris.MODE_DENSE, 1.0, [0])
    assert mask.info().dense == 1
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=13, outliers=True)
    ref_pool = ris.ris_attention_masked(mask, q, k, v, rope=rope)
    spec = ora.MaskSpec(N=N, mode=ora.MODE_DENSE, density=1.0, seeds=[0])
    o_ref, lse_ref, _, _ = ora.sparse_attention(qn, kn, vn, spec, oracle_rope(3, 1e6, 256))
    for _ in range(2):
        out = torch.full((N, Hq, D), float("nan"), dtype=torch.bfloat16, device="cuda")
        lse = torch.empty((Hq, N), dtype=torch.float32, device="cuda")
        ris.ris_attention_masked_noalloc(mask, q, k, v, out, rope=rope, lse=lse)
        torch.cuda.synchronize()
        check_bf16_path(to_np(out), o_ref, out_bf16=True)
        np.testing.assert_allclose(to_np(lse).T, lse_ref, rtol=0, atol=2e-3)
        # against the pool path: each bf16 output is within half an ulp of its fp32 value
        diff = np.abs(to_np(out) - to_np(ref_pool))
        assert np.all(diff <= BF16_MAX_ABS + 2.0 ** -7 * np.abs(to_np(ref_pool)))
    mask.free()


def test_noalloc_structural_blocks_against_oracle():
    """A Structural mask with blocks of 300 tokens (ris_attention_masked takes the dense-suffix
    split) on the gather alone, against the oracle."""
    N, Hq, Hkv, D = 3000, 6, 2, 128
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 256)
    mask = ris.ris_mask_generate(N, Hkv, ris.MODE_STRUCTURAL, 0.1, [4])
    assert ris.ris_attention_design(mask, torch.bfloat16, D) == 4
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=29, outliers=True)
    out = torch.empty((N, Hq, D), dtype=torch.float32, device="cuda")
    ris.ris_attention_masked_noalloc(mask, q, k, v, out, rope=rope)
    torch.cuda.synchronize()
    spec = ora.MaskSpec(N=N, mode=ora.MODE_STRUCTURAL, density=0.1, seeds=[4])
    o_ref, _, _, _ = ora.sparse_attention(qn, kn, vn, spec, oracle_rope(3, 1e6, 256))
    check_bf16_path(to_np(out), o_ref)
    mask.free()


def test_noalloc_without_rope_and_per_seed():
    N, Hq, Hkv, D = 1500, 6, 2, 128
    mask = ris.ris_mask_generate(N, Hkv, 0, 0.05, [4, 5], per_seed=True)
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=21, outliers=True)
    ref = ris.ris_attention_masked(mask, q, k, v, out_dtype=torch.float32)
    for _ in range(2):
        out = torch.empty((2, N, Hq, D), dtype=torch.float32, device="cuda")
        ris.ris_attention_masked_noalloc(mask, q, k, v, out)
        torch.cuda.synchronize()
        _compare(out, ref, False)
    mask.free()


def test_noalloc_refuses_sizes_beyond_its_scratch_and_wide_groups():
    N, Hq, Hkv, D = 16384, 12, 2, 128  # needs 7168 B per token > 64 MiB in total
    mask = ris.ris_mask_generate(N, Hkv, 0, 0.001, [0])
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=3)
    out = torch.zeros((N, Hq, D), dtype=torch.bfloat16, device="cuda")
    n0 = ris.ris_launch_count()
    with pytest.raises(ris.RisError) as e:
        ris.ris_attention_masked_noalloc(mask, q, k, v, out, rope=ris.rope_cfg(ris.ROPE_PLAIN, 1e6, 32768))
    assert e.value.status == ris.RIS_ERR_INVALID and "at most" in str(e.value)
    assert ris.ris_launch_count() == n0
    torch.cuda.synchronize()
    assert not out.any()
    mask.free()
    N, Hq, Hkv = 300, 16, 1  # 16 query heads per KV head: only the tiles take them
    mask = ris.ris_mask_generate(N, Hkv, 0, 0.05, [0])
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=3)
    out = torch.zeros((N, Hq, D), dtype=torch.bfloat16, device="cuda")
    n0 = ris.ris_launch_count()
    with pytest.raises(ris.RisError) as e:
        ris.ris_attention_masked_noalloc(mask, q, k, v, out)
    assert e.value.status == ris.RIS_ERR_UNSUPPORTED
    assert ris.ris_launch_count() == n0
    mask.free()
