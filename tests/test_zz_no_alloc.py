"""The allocation-free layer entry point, ris_attention_masked_noalloc, through the C ABI.

It serves callers that may not allocate device memory while a layer runs (an inference
engine's enqueue callback, a server with a memory plan fixed at load time). Its results must
match ris_attention_masked's within the parity tolerance, on consecutive calls that reuse the
same fixed scratch array, and sizes beyond that array must be refused before any launch.
This file is collected last so that a failure here never hides the other GPU tests.
"""
import numpy as np
import pytest
import torch

from helpers import BF16_MAX_ABS, BF16_REL_L2, F32_REL_L2, make_inputs, rel_l2, to_np
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def _compare(got, ref, fp32):
    g, r = to_np(got), to_np(ref)
    if fp32:
        assert rel_l2(g, r) <= F32_REL_L2
    else:
        assert np.abs(g - r).max() <= BF16_MAX_ABS and rel_l2(g, r) <= BF16_REL_L2


@pytest.mark.parametrize("dtype,Hq,Hkv,D,mode", [(torch.bfloat16, 12, 2, 128, 0), (torch.float32, 4, 1, 64, 1)])
def test_noalloc_matches_pool_path_on_consecutive_calls(dtype, Hq, Hkv, D, mode):
    N = 3000
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 1024)
    mask = ris.ris_mask_generate(N, Hkv, mode, 0.03, [0, 1, 2])
    fp32 = dtype == torch.float32
    for call, seed in enumerate((11, 12)):  # two calls in a row, different inputs
        (q, k, v), _ = make_inputs(N, Hq, Hkv, D, dtype=dtype, seed=seed, outliers=not fp32)
        ref = ris.ris_attention_masked(mask, q, k, v, rope=rope, out_dtype=torch.float32)
        out = torch.full((N, Hq, D), float("nan"), dtype=torch.float32, device="cuda")
        lse = torch.empty((Hq, N), dtype=torch.float32, device="cuda")
        ris.ris_attention_masked_noalloc(mask, q, k, v, out, rope=rope, lse=lse)
        torch.cuda.synchronize()
        assert torch.isfinite(out).all(), f"call {call}"
        _compare(out, ref, fp32)
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


def test_noalloc_refuses_sizes_beyond_its_scratch():
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
