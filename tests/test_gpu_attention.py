"""GPU RoPE and sparse attention vs the fp64 oracle, through the C ABI.

Tolerances (see helpers.py): bf16 inputs with fp32 accumulation must be within max-abs
1e-2 and relative L2 5e-3 of the fp64 oracle; fp32 inputs within relative L2 1e-5.
Small cases compare every output; the full workload sizes compare sampled rows, computed
one by one by the oracle, in the same launch configuration the benchmark uses.
"""
import numpy as np
import pytest
import torch

import oracle as ora
from helpers import (check_bf16_path, check_f32_path, make_inputs, oracle_rope, rel_l2, sample_rows,
                     to_np)
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu

QWEN = dict(Hq=12, Hkv=2, D=128, theta=1e6, native=32768)
TINY = dict(Hq=32, Hkv=4, D=64, theta=1e4, native=2048)


def run_gpu(q, k, v, mode, d, seeds, rope_kind, theta, native, out_dtype=torch.float32, opts=None,
            per_seed=False, return_lse=True):
    rope = ris.rope_cfg(rope_kind, theta, native) if rope_kind else None
    fn = ris.ris_ensemble_batch if per_seed else ris.ris_sparse_attention_fwd
    out, lse = fn(q, k, v, mode, d, seeds, rope=rope, opts=opts, out_dtype=out_dtype, return_lse=True)
    torch.cuda.synchronize()
    return out, lse


def run_oracle(qn, kn, vn, mode, d, seeds, rope_kind, theta, native, rows=None, seed_index=-1, W=1, A=0,
               head_key=0, sampler=0):
    N = qn.shape[0]
    spec = ora.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, seed_index=seed_index, local_window=W,
                        n_anchor=A, head_key=head_key, sampler=sampler)
    out, lse, _, _ = ora.sparse_attention(qn, kn, vn, spec, oracle_rope(rope_kind, theta, native), rows=rows)
    return out, lse


# ----------------------------------------------------------------------------- RoPE
@pytest.mark.parametrize("kind,N,native", [(1, 300, 4096), (2, 1024, 256), (3, 4096, 1024), (3, 65536, 32768)])
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_rope_apply(kind, N, native, dtype):
    H, D, theta = 3, 128, 1e6
    (x, _, _), (xn, _, _) = make_inputs(N, H, 1, D, dtype=dtype, seed=kind)
    ris.ris_rope_apply(x, ris.rope_cfg(kind, theta, native))
    torch.cuda.synchronize()
    ref = ora.rope(xn, np.arange(N, dtype=np.float64), ora.RopeCfg(kind=kind, theta=theta, native_len=native), N)
    got = to_np(x)
    if dtype == torch.float32:
        # fp32 rotation of exactly reduced angles: a few ulps of the largest pair element
        assert np.abs(got - ref).max() <= 4e-6 * max(1.0, np.abs(ref).max())
    else:
        # bf16 result: one bf16 ulp of the exact rotation, plus the fp32 rotation's own error
        # (a few fp32 ulps of the pair's inputs) for outputs that cancel to almost zero
        ulp = 2.0 ** (np.floor(np.log2(np.maximum(np.abs(ref), 1e-30))) - 7)
        pair = np.concatenate([np.maximum(np.abs(xn[..., :D // 2]), np.abs(xn[..., D // 2:]))] * 2, -1)
        assert np.all(np.abs(got - ref) <= ulp + 4e-7 * pair * 1.07)


# ----------------------------------------------------------------------------- small, full outputs
SMALL = [
    # N, Hq, Hkv, D, dtype, mode, d, S, rope kind, native
    (1, 1, 1, 128, torch.float32, 0, 0.05, 1, 1, 4096),
    (33, 4, 2, 64, torch.bfloat16, 0, 0.3, 2, 0, 4096),
    (200, 6, 2, 128, torch.bfloat16, 1, 0.05, 3, 2, 64),
    (517, 8, 1, 64, torch.bfloat16, 0, 0.05, 5, 3, 128),
    (640, 3, 3, 128, torch.float32, 1, 0.1, 2, 3, 128),
    (300, 12, 2, 128, torch.bfloat16, 2, 1.0, 1, 1, 4096),
    (300, 2, 1, 64, torch.float32, 0, 1.0, 1, 0, 4096),
    (1025, 5, 1, 128, torch.bfloat16, 0, 0.02, 10, 1, 4096),
    # tiny and ragged sizes on the tile design (their masks keep most causal pairs)
    (1, 6, 2, 128, torch.bfloat16, 0, 0.05, 1, 3, 64),
    (2, 6, 2, 128, torch.bfloat16, 1, 0.5, 2, 1, 4096),
    (129, 12, 2, 128, torch.bfloat16, 0, 0.3, 3, 3, 64),
    (257, 6, 2, 128, torch.bfloat16, 2, 1.0, 1, 3, 64),
    (130, 6, 2, 128, torch.bfloat16, 0, 0.01, 1, 1, 4096),
    # the register gather's fp8 form (rotated bf16, head dim 128) at 1, 5 and 8 query heads per
    # KV head: every head of the tensor-core tile's N dimension used, or some left empty
    (700, 2, 2, 128, torch.bfloat16, 1, 0.01, 2, 1, 4096),
    (901, 5, 1, 128, torch.bfloat16, 0, 0.03, 1, 3, 256),
    (700, 8, 1, 128, torch.bfloat16, 0, 0.02, 1, 3, 256),
]


@pytest.mark.parametrize("N,Hq,Hkv,D,dtype,mode,d,S,kind,native", SMALL)
def test_attention_small_full(N, Hq, Hkv, D, dtype, mode, d, S, kind, native):
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, dtype=dtype, seed=N + S, outliers=(dtype == torch.bfloat16))
    seeds = list(range(S))
    out, lse = run_gpu(q, k, v, mode, d, seeds, kind, 1e4, native)
    ref, ref_lse = run_oracle(qn, kn, vn, mode, d, seeds, kind, 1e4, native)
    if dtype == torch.float32:
        check_f32_path(to_np(out), ref)
        np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=1e-5, atol=1e-5)
    else:
        check_bf16_path(to_np(out), ref)
        np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-2)


def test_attention_bf16_output_and_forced_set():
    N, Hq, Hkv, D = 700, 6, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=7, outliers=True)
    opts = ris.mask_opts(local_window=16, n_anchor=4)
    out = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.02, [1, 2], rope=ris.rope_cfg(1, 1e6, 32768), opts=opts)
    torch.cuda.synchronize()
    assert out.dtype == torch.bfloat16
    ref, _ = run_oracle(qn, kn, vn, 0, 0.02, [1, 2], 1, 1e6, 32768, W=16, A=4)
    check_bf16_path(to_np(out), ref, out_bf16=True)


@pytest.mark.parametrize("mode", [0, 1], ids=["stochastic", "structural"])
def test_attention_index_draw_sampler(mode):
    """The whole path on a mask from the index-draw sampler (torch.randint reading)."""
    N, Hq, Hkv, D = 900, 6, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=11, outliers=True)
    opts = ris.mask_opts(sampler=ris.SAMPLER_DRAWS)
    out, lse = run_gpu(q, k, v, mode, 0.03, [4, 5, 6], 3, 1e6, 256, opts=opts)
    ref, ref_lse = run_oracle(qn, kn, vn, mode, 0.03, [4, 5, 6], 3, 1e6, 256, sampler=1)
    check_bf16_path(to_np(out), ref)
    np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-2)


def test_attention_per_head_masks():
    N, Hq, Hkv, D = 400, 8, 2, 64
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=11)
    opts = ris.mask_opts(per_head=True)
    out = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.1, [4], opts=opts, out_dtype=torch.float32)
    torch.cuda.synchronize()
    got = to_np(out)
    G = Hq // Hkv
    for g in range(Hkv):
        ref, _ = run_oracle(qn[:, g * G:(g + 1) * G], kn[:, g:g + 1], vn[:, g:g + 1], 0, 0.1, [4], 0, 1e4, 4096,
                            head_key=g)
        check_bf16_path(got[:, g * G:(g + 1) * G], ref)


def test_ensemble_batch_small_full():
    N, Hq, Hkv, D, seeds = 600, 6, 2, 128, [3, 4, 5, 6]
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=5, outliers=True)
    out, lse = run_gpu(q, k, v, 0, 0.05, seeds, 1, 1e6, 32768, per_seed=True)
    assert out.shape == (4, N, Hq, D)
    for s in range(len(seeds)):
        ref, ref_lse = run_oracle(qn, kn, vn, 0, 0.05, seeds, 1, 1e6, 32768, seed_index=s)
        check_bf16_path(to_np(out[s]), ref)
        np.testing.assert_allclose(to_np(lse[s]).T, ref_lse, rtol=0, atol=2e-2)


def test_attention_masked_reuses_mask_across_layers():
    N, Hq, Hkv, D = 512, 12, 2, 128
    m = ris.ris_mask_generate(N, Hkv, 1, 0.05, [1, 2, 3])
    rope = ris.rope_cfg(3, 1e6, 256)
    for layer in range(3):
        (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=100 + layer, outliers=True)
        out = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
        torch.cuda.synchronize()
        ref, _ = run_oracle(qn, kn, vn, 1, 0.05, [1, 2, 3], 3, 1e6, 256)
        check_bf16_path(to_np(out), ref)
    m.free()


def test_v_constant_gives_one():
    N, Hq, Hkv, D = 1000, 6, 2, 128
    (q, k, _), _ = make_inputs(N, Hq, Hkv, D, seed=2, outliers=True)
    v = torch.ones(N, Hkv, D, dtype=torch.bfloat16, device="cuda")
    out = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.05, [0, 1], out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.all((out - 1).abs() < 1e-5)


# ----------------------------------------------------------------------------- workload configurations
def _config_case(N, shape, dtype, mode, d, S, kind, outliers, nrows, seed=0, per_seed=False, opts=None):
    (q, k, v), (qn, kn, vn) = make_inputs(N, shape["Hq"], shape["Hkv"], shape["D"], dtype=dtype, seed=seed,
                                          outliers=outliers)
    seeds = list(range(S))
    out, lse = run_gpu(q, k, v, mode, d, seeds, kind, shape["theta"], shape["native"], per_seed=per_seed,
                       opts=opts)
    rows = np.arange(N) if nrows is None else sample_rows(N, nrows, seed=N + S)
    got = to_np(out[rows] if not per_seed else out[:, rows])
    return got, (qn, kn, vn), seeds, rows, to_np(lse)


def test_c1_single_head_fp32_full():
    """N=2048, 1 head, D=128, fp32, theta 1e6, Stochastic 5%, 1 seed; every output."""
    shape = dict(Hq=1, Hkv=1, D=128, theta=1e6, native=32768)
    got, (qn, kn, vn), seeds, rows, lse = _config_case(2048, shape, torch.float32, 0, 0.05, 1, 1, False, None)
    ref, ref_lse = run_oracle(qn, kn, vn, 0, 0.05, seeds, 1, 1e6, 32768)
    check_f32_path(got, ref)
    np.testing.assert_allclose(lse.T, ref_lse, rtol=1e-6, atol=1e-6)


def test_c2_qwen_8k_full():
    """Qwen2 shape, N=8192, bf16 with outlier channels, Stochastic 1% x 10 seeds; every output."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(8192, QWEN, torch.bfloat16, 0, 0.01, 10, 1, True, None)
    ref, _ = run_oracle(qn, kn, vn, 0, 0.01, seeds, 1, 1e6, 32768)
    check_bf16_path(got, ref)


def test_c3_tinyllama_16k_yarn_structural():
    """TinyLlama shape, N=16384 (YaRN s=8 beyond the 2048 window), Structural 1% x 10; sampled rows."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(16384, TINY, torch.bfloat16, 1, 0.01, 10, 3, False, 384)
    ref, _ = run_oracle(qn, kn, vn, 1, 0.01, seeds, 3, 1e4, 2048, rows=rows)
    check_bf16_path(got, ref)


@pytest.mark.parametrize("mode,d,S", [(0, 0.01, 70), (0, 0.05, 10), (2, 1.0, 1)], ids=["1pct_x70", "5pct_x10", "dense"])
def test_c4_qwen_32k(mode, d, S):
    """Qwen2 shape, N=32768, bf16 with outliers: Stochastic 1% x 70, 5% x 10 and dense causal; sampled rows."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(32768, QWEN, torch.bfloat16, mode, d, S, 1, True, 96)
    ref, _ = run_oracle(qn, kn, vn, mode, d, seeds, 1, 1e6, 32768, rows=rows)
    check_bf16_path(got, ref)


@pytest.mark.parametrize("mode", [0, 1], ids=["stochastic", "structural"])
def test_c5_qwen_64k_layer(mode):
    """One layer of the N=65536 stack (YaRN s=2), 1% x 10 seeds; about 1024 sampled rows."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(65536, QWEN, torch.bfloat16, mode, 0.01, 10, 3, True, 1024,
                                                     seed=3)
    assert rows.shape[0] >= 1000  # first, last and ~1024 random rows, all heads
    ref, _ = run_oracle(qn, kn, vn, mode, 0.01, seeds, 3, 1e6, 32768, rows=rows)
    check_bf16_path(got, ref)


@pytest.mark.parametrize("mode", [0, 1], ids=["stochastic", "structural"])
def test_c6_paper_geometry_64k_layer(mode):
    """The N=65536 layer with the paper's geometry (local window 1024 + 4 anchors); sampled rows."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(65536, QWEN, torch.bfloat16, mode, 0.01, 10, 3, True, 64,
                                                     seed=5, opts=ris.paper_geometry())
    ref, _ = run_oracle(qn, kn, vn, mode, 0.01, seeds, 3, 1e6, 32768, rows=rows, W=ris.PRESET_LOCAL_WINDOW,
                        A=ris.PRESET_ANCHORS)
    check_bf16_path(got, ref)


def test_c5_ensemble_per_seed_sampled():
    """Per-seed ensemble at N=65536 (YaRN s=2, 10 seeds in one launch): sampled rows of three seeds."""
    got, (qn, kn, vn), seeds, rows, _ = _config_case(65536, QWEN, torch.bfloat16, 0, 0.01, 10, 3, True, 24,
                                                     seed=4, per_seed=True)
    for s in (0, 5, 9):
        ref, _ = run_oracle(qn, kn, vn, 0, 0.01, seeds, 3, 1e6, 32768, rows=rows, seed_index=s)
        check_bf16_path(got[s], ref)


def test_c2_ensemble_per_seed_sampled():
    got, (qn, kn, vn), seeds, rows, _ = _config_case(8192, QWEN, torch.bfloat16, 0, 0.01, 10, 1, True, 64,
                                                     per_seed=True)
    for s in (0, 9):
        ref, _ = run_oracle(qn, kn, vn, 0, 0.01, seeds, 1, 1e6, 32768, rows=rows, seed_index=s)
        check_bf16_path(got[s], ref)


def test_attention_u32_keys_beyond_65536():
    """N > 65536 stores 32-bit key indices; sampled rows against the oracle."""
    N, Hq, Hkv, D = 65600, 2, 1, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=17, outliers=True)
    out = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.0005, [2], rope=ris.rope_cfg(3, 1e6, 32768),
                                       out_dtype=torch.float32)
    torch.cuda.synchronize()
    rows = sample_rows(N, 24, seed=5)
    ref, _ = run_oracle(qn, kn, vn, 0, 0.0005, [2], 3, 1e6, 32768, rows=rows)
    check_bf16_path(to_np(out[rows]), ref)


def test_dense_tiles_bf16_output_and_lse():
    """High union density goes to the masked-tile kernel; bf16 output and lse against the oracle."""
    N, Hq, Hkv, D = 600, 12, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=23, outliers=True)
    out, lse = ris.ris_sparse_attention_fwd(q, k, v, 0, 0.5, [1, 2], rope=ris.rope_cfg(3, 1e6, 256),
                                            return_lse=True)
    torch.cuda.synchronize()
    ris.ris_device_status()
    ref, ref_lse = run_oracle(qn, kn, vn, 0, 0.5, [1, 2], 3, 1e6, 256)
    check_bf16_path(to_np(out), ref, out_bf16=True)
    np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-2)


@pytest.mark.parametrize("d,S,D", [(0.02, 3, 128), (0.5, 2, 128), (1.0, 1, 128), (0.03, 2, 64)],
                         ids=["gather", "tiles", "dense", "hd64"])
def test_row_ranges_reassemble_the_layer(d, S, D):
    """Balanced row ranges computed one call each reassemble the whole-layer output bit for bit
    (gather and tile designs, ranges that cut through 128-row tiles)."""
    N, Hq, Hkv = 1500, 6, 2
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=17, outliers=True)
    mode = 2 if d >= 1.0 else 0
    m = ris.ris_mask_generate(N, Hkv, mode, d, list(range(S)))
    rope = ris.rope_cfg(3, 1e6, 256)
    whole = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
    bounds = ris.ris_mask_row_split(m, 3)
    assert bounds[0] == 0 and bounds[-1] == N and sorted(set(bounds)) == bounds
    parts = torch.full_like(whole, float("nan"))
    for r0, r1 in zip(bounds[:-1], bounds[1:]):
        ris.ris_attention_masked_rows(m, r0, r1, q, k, v, parts, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(parts, whole)
    one = torch.full_like(whole, float("nan"))
    ris.ris_attention_masked_rows(m, 700, 701, q, k, v, one, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(one[700], whole[700]) and torch.isnan(one[:700]).all() and torch.isnan(one[701:]).all()
    with pytest.raises(ris.RisError):
        ris.ris_attention_masked_rows(m, 5, 5, q, k, v, one, rope=rope)
    m.free()


def test_structural_split_design_choice():
    """C5's Structural mask (blocks of 655) takes the dense-suffix split: cliques on the tiles,
    the rest gathered, at head_dim 128 and 64; Structural masks with small blocks and no wide
    window, and per-seed masks, do not; a Stochastic mask with a 1024-key window does."""
    m = ris.ris_mask_generate(65536, 2, 1, 0.01, list(range(10)))
    assert ris.ris_attention_design(m, torch.bfloat16, 128) == 4
    assert ris.ris_attention_design(m, torch.bfloat16, 64) == 4
    m.free()
    m = ris.ris_mask_generate(2000, 2, 1, 0.05, [1])  # B = min(200, 100) = 100 < 256
    assert ris.ris_attention_design(m, torch.bfloat16, 128) in (0, 2)
    m.free()
    m = ris.ris_mask_generate(65536, 2, 1, 0.01, list(range(10)), per_seed=True)
    assert ris.ris_attention_design(m, torch.bfloat16, 128) != 4
    m.free()
    m = ris.ris_mask_generate(65536, 2, 0, 0.005, list(range(4)), opts=ris.paper_geometry())
    assert ris.ris_attention_design(m, torch.bfloat16, 128) == 4
    m.free()


@pytest.mark.parametrize("N,mode,d,S,kind,window,anchors", [
    (3000, 1, 0.1, 1, 3, 1, 0), (2700, 1, 0.11, 1, 0, 1, 0), (4100, 1, 0.08, 1, 3, 40, 3),
    (3300, 1, 0.1, 1, 3, 700, 2), (2900, 0, 0.01, 2, 3, 300, 4), (1500, 1, 0.002, 1, 3, 600, 0),
    (2560, 1, 0.1, 1, 3, 1, 0), (1000, 0, 0.02, 1, 3, 256, 0), (700, 0, 0.02, 1, 0, 900, 0)],
    ids=["blocks", "blocks_pre_rotated", "blocks_small_window_anchors", "blocks_in_wider_window",
         "stochastic_window", "structural_small_blocks_window", "blocks_of_exactly_256",
         "window_of_exactly_256", "window_longer_than_the_sequence"])
def test_dense_suffix_split_full(N, mode, d, S, kind, window, anchors):
    """The dense-suffix split (Structural blocks of >= 256 tokens and / or a local window of
    >= 256 keys on the tiles, the other keys gathered) against the oracle on every row: fp32
    and bf16 outputs and the log-sum-exp, with and without RoPE, with anchors and with windows
    shorter and longer than the blocks."""
    Hq, Hkv, D = 12, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=N, outliers=True)
    seeds = list(range(5, 5 + S))
    opts = ris.mask_opts(local_window=window, n_anchor=anchors)
    m = ris.ris_mask_generate(N, Hkv, mode, d, seeds, opts=opts)
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 4
    rope = ris.rope_cfg(kind, 1e6, 256) if kind else None
    out32, lse = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32, return_lse=True)
    out16 = ris.ris_attention_masked(m, q, k, v, rope=rope)
    torch.cuda.synchronize()
    ris.ris_device_status()
    m.free()
    ref, ref_lse = run_oracle(qn, kn, vn, mode, d, seeds, kind, 1e6, 256, W=window, A=anchors)
    check_bf16_path(to_np(out32), ref)
    check_bf16_path(to_np(out16), ref, out_bf16=True)
    np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-3)


def test_structural_split_row_ranges():
    """Row ranges through the dense-suffix split reassemble the whole layer bit for bit."""
    N, Hq, Hkv, D = 3000, 6, 2, 128
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=29, outliers=True)
    m = ris.ris_mask_generate(N, Hkv, 1, 0.1, [4])
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 4
    rope = ris.rope_cfg(3, 1e6, 256)
    whole = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
    bounds = ris.ris_mask_row_split(m, 4)
    parts = torch.full_like(whole, float("nan"))
    for r0, r1 in zip(bounds[:-1], bounds[1:]):
        ris.ris_attention_masked_rows(m, r0, r1, q, k, v, parts, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(parts, whole)
    m.free()


def test_dense_suffix_split_per_head_masks():
    """Per-head masks (keyed per KV head) take the dense-suffix split too: each KV head
    gathers from its own key lists after the shared suffix pass."""
    N, Hq, Hkv, D = 2800, 6, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=31, outliers=True)
    opts = ris.mask_opts(per_head=True, local_window=300)
    m = ris.ris_mask_generate(N, Hkv, 1, 0.1, [2], opts=opts)
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 4
    out = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e6, 256), out_dtype=torch.float32)
    torch.cuda.synchronize()
    m.free()
    G = Hq // Hkv
    for g in range(Hkv):
        spec = ora.MaskSpec(N=N, mode=1, density=0.1, seeds=[2], local_window=300, head_key=g)
        ref, _, _, _ = ora.sparse_attention(qn[:, g * G:(g + 1) * G], kn[:, g:g + 1], vn[:, g:g + 1], spec,
                                            oracle_rope(3, 1e6, 256))
        check_bf16_path(to_np(out[:, g * G:(g + 1) * G]), ref)


def test_dense_suffix_split_u32_keys_beyond_65536():
    """N > 65536 (32-bit key lists) with Structural blocks of 656 tokens: the split on sampled rows."""
    N, Hq, Hkv, D = 65600, 2, 1, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=19, outliers=True)
    m = ris.ris_mask_generate(N, Hkv, 1, 0.01, [1, 2])
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 4
    out = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e6, 32768), out_dtype=torch.float32)
    torch.cuda.synchronize()
    m.free()
    rows = sample_rows(N, 24, seed=7)
    ref, _ = run_oracle(qn, kn, vn, 1, 0.01, [1, 2], 3, 1e6, 32768, rows=rows)
    check_bf16_path(to_np(out[rows]), ref)


@pytest.mark.parametrize("mode,d,S", [(0, 0.01, 4), (1, 0.01, 2), (0, 0.01, 12)], ids=["stochastic_gather", "structural_split", "stochastic_tiles"])
def test_quarter_million_tokens_sampled(mode, d, S):
    """N = 262144 (bitmap of 4.3 GB, byte offsets past 2^32, 32-bit key lists; 256 K keys per
    row at most): sampled rows of the gather, the dense-suffix split and the tile design."""
    N, Hq, Hkv, D = 262144, 2, 1, 128
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=41, outliers=True)
    seeds = list(range(S))
    m = ris.ris_mask_generate(N, Hkv, mode, d, seeds)
    design = ris.ris_attention_design(m, torch.bfloat16, D)
    assert design == {"stochastic_gather": 0, "structural_split": 4, "stochastic_tiles": 2}[
        {(0, 4): "stochastic_gather", (1, 2): "structural_split", (0, 12): "stochastic_tiles"}[(mode, S)]]
    out = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e6, 32768), out_dtype=torch.float32)
    torch.cuda.synchronize()
    ris.ris_device_status()
    m.free()
    rows = sample_rows(N, 12, seed=3)
    ref, _ = run_oracle(qn, kn, vn, mode, d, seeds, 3, 1e6, 32768, rows=rows)
    check_bf16_path(to_np(out[rows]), ref)


def test_row_ranges_per_seed_sets():
    """Row ranges of a per-seed mask (one output set per seed, walked by the gather's set loop)
    reassemble the whole per-seed output bit for bit."""
    N, Hq, Hkv, D, seeds = 1400, 6, 2, 128, [3, 4, 5]
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=37, outliers=True)
    m = ris.ris_mask_generate(N, Hkv, 0, 0.03, seeds, per_seed=True)
    assert ris.ris_attention_design(m, torch.bfloat16, D) == 0
    rope = ris.rope_cfg(3, 1e6, 256)
    whole = torch.empty(len(seeds), N, Hq, D, dtype=torch.float32, device="cuda")
    ris.ris_attention_masked_rows(m, 0, N, q, k, v, whole, rope=rope)
    parts = torch.full_like(whole, float("nan"))
    for r0, r1 in ((0, 333), (333, 900), (900, 1399), (1399, 1400)):
        ris.ris_attention_masked_rows(m, r0, r1, q, k, v, parts, rope=rope)
    torch.cuda.synchronize()
    assert torch.equal(parts, whole)
    ref = ris.ris_ensemble_batch(q, k, v, 0, 0.03, seeds, rope=rope, out_dtype=torch.float32)
    torch.cuda.synchronize()
    assert torch.equal(ref, whole)
    m.free()


@pytest.mark.parametrize("Hq,Hkv,D,d,S", [(16, 1, 128, 0.02, 2), (24, 2, 128, 0.3, 1), (16, 1, 64, 0.05, 1)],
                         ids=["mqa_16_sparse", "group_12", "mqa_16_hd64"])
def test_groups_wider_than_eight_on_tiles(Hq, Hkv, D, d, S):
    """More than 8 query heads per KV head (multi-query attention): bf16 runs on the tile
    design whatever the density; fp32 reports RIS_ERR_UNSUPPORTED."""
    N = 700
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=43, outliers=True)
    seeds = list(range(S))
    out, lse = ris.ris_sparse_attention_fwd(q, k, v, 0, d, seeds, rope=ris.rope_cfg(3, 1e6, 256),
                                            out_dtype=torch.float32, return_lse=True)
    torch.cuda.synchronize()
    ris.ris_device_status()
    ref, ref_lse = run_oracle(qn, kn, vn, 0, d, seeds, 3, 1e6, 256)
    check_bf16_path(to_np(out), ref)
    np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-3)
    with pytest.raises(ris.RisError):
        ris.ris_sparse_attention_fwd(q.float(), k.float(), v.float(), 0, d, seeds, out_dtype=torch.float32)


@pytest.mark.parametrize("N,mode,d,S,W,Hq,Hkv,design", [
    (1100, 0, 0.3, 2, 1, 32, 4, 2), (900, 2, 1.0, 1, 1, 8, 1, 2), (3000, 1, 0.1, 1, 1, 32, 4, 4),
    (2000, 0, 0.01, 1, 400, 16, 2, 4)], ids=["tiles", "dense", "suffix_split_blocks", "suffix_split_window"])
def test_head_dim_64_on_tiles(N, mode, d, S, W, Hq, Hkv, design):
    """head_dim 64 (TinyLlama-shaped heads) on the tile design and the dense-suffix split,
    every row against the oracle, with the log-sum-exp."""
    D = 64
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=N + 1, outliers=True)
    seeds = list(range(S))
    m = ris.ris_mask_generate(N, Hkv, mode, d, seeds, opts=ris.mask_opts(local_window=W))
    assert ris.ris_attention_design(m, torch.bfloat16, D) == design
    out, lse = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e4, 256), out_dtype=torch.float32,
                                        return_lse=True)
    torch.cuda.synchronize()
    ris.ris_device_status()
    m.free()
    ref, ref_lse = run_oracle(qn, kn, vn, mode, d, seeds, 3, 1e4, 256, W=W)
    check_bf16_path(to_np(out), ref)
    np.testing.assert_allclose(to_np(lse).T, ref_lse, rtol=0, atol=2e-3)


@pytest.mark.parametrize("N,mode,d,S,layer", [
    (32768, 0, 0.01, 70, 0), (65536, 0, 0.01, 10, 7), (65536, 1, 0.01, 10, 7), (65536, 0, 0.01, 70, 27),
    (65536, 1, 0.01, 70, 27)],
    ids=["c4a_32k_1pct_x70", "c5_64k_stochastic_x10", "c5_64k_structural_x10", "c5_64k_stochastic_x70",
         "c5_64k_structural_x70"])
def test_benchmarked_layers_bf16_output(N, mode, d, S, layer):
    """The layers the benchmark times, in its own configuration: a mask built once and
    ris_attention_masked with bf16 outputs (the bench's output dtype), YaRN with native window
    32768, inputs of the layer's seed; about 1024 sampled rows (all heads) against the oracle.
    Covers the 65,536-token 70-seed run in both modes (Results, "Ensemble Coverage Analysis")."""
    (q, k, v), (qn, kn, vn) = make_inputs(N, QWEN["Hq"], QWEN["Hkv"], QWEN["D"], seed=layer, outliers=True)
    seeds = list(range(S))
    m = ris.ris_mask_generate(N, QWEN["Hkv"], mode, d, seeds)
    design = ris.ris_attention_design(m, torch.bfloat16, QWEN["D"])
    out = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e6, 32768))
    torch.cuda.synchronize()
    ris.ris_device_status()
    m.free()
    assert out.dtype == torch.bfloat16
    rows = sample_rows(N, 1024, seed=N + S + mode)
    assert rows.shape[0] >= 1000
    ref, _ = run_oracle(qn, kn, vn, mode, d, seeds, 3, 1e6, 32768, rows=rows)
    err, rel = check_bf16_path(to_np(out[rows]), ref, out_bf16=True)
    print(f"design {design}: max-abs {err:.2e}, rel-L2 {rel:.2e}")


@pytest.mark.parametrize("mode,d,S,W", [(0, 0.02, 3, 1), (0, 0.5, 2, 1), (2, 1.0, 1, 1), (1, 0.1, 1, 1), (0, 0.01, 1, 300)],
                         ids=["gather", "tiles", "dense", "suffix_split_blocks", "suffix_split_window"])
def test_local_row_shards_reassemble_the_layer(mode, d, S, W):
    """The row-sharded prefill with K/V all-gather, its ranks run one after the other on one
    GPU: every rank holds only its rows of q (and gets the whole K and V, as the all-gather
    returns them), calls ris_attention_masked_local, and the parts reassemble the whole-layer
    output and log-sum-exp bit for bit, in every design."""
    N, Hq, Hkv, D = 1700, 6, 2, 128
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=53, outliers=True)
    m = ris.ris_mask_generate(N, Hkv, mode, d, list(range(S)), opts=ris.mask_opts(local_window=W))
    rope = ris.rope_cfg(3, 1e6, 256)
    whole, lse = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32, return_lse=True)
    b = ris.ris_mask_row_split(m, 3)
    parts, lparts = [], []
    for r in range(3):
        o, l = ris.ris_attention_masked_local(m, b[r], b[r + 1], q[b[r]:b[r + 1]].clone(), k, v, rope=rope,
                                              out_dtype=torch.float32, return_lse=True)
        parts.append(o)
        lparts.append(l)
    torch.cuda.synchronize()
    ris.ris_device_status()
    assert torch.equal(torch.cat(parts, 0), whole)
    assert torch.equal(torch.cat(lparts, 1), lse)
    # without RoPE (q and k used as given) and bf16 outputs
    whole16 = ris.ris_attention_masked(m, q, k, v)
    part = ris.ris_attention_masked_local(m, b[1], b[2], q[b[1]:b[2]].clone(), k, v)
    torch.cuda.synchronize()
    assert torch.equal(part, whole16[b[1]:b[2]])
    m.free()


def test_local_rows_refuse_per_seed_masks():
    N, Hq, Hkv, D = 300, 6, 2, 128
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=5)
    m = ris.ris_mask_generate(N, Hkv, 0, 0.05, [1, 2], per_seed=True)
    with pytest.raises(ris.RisError) as e:
        ris.ris_attention_masked_local(m, 0, 100, q[:100].clone(), k, v)
    assert e.value.status == ris.RIS_ERR_UNSUPPORTED
    m.free()


@pytest.mark.parametrize("scale_exp", [14, 20])
def test_tile_values_beyond_fp16_range(scale_exp):
    """The tile kernel takes the values as fp16 scaled by a power of two chosen from their
    largest magnitude (none below 2^14). Values scaled by 2^14 and 2^20 (beyond fp16's 65504)
    must give exactly that multiple of the unscaled output (the scale is a power of two, so
    every operand and the fp32 accumulation scale exactly), within the parity tolerance of the
    oracle once divided back, for the tiles, the dense mode and the dense-suffix split."""
    N, Hq, Hkv, D = 3000, 6, 2, 128  # Structural blocks of 300 tokens: the dense-suffix split
    (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=61, outliers=True)
    big = v * (2.0 ** scale_exp)
    rope = ris.rope_cfg(3, 1e6, 256)
    for mode, d, S, design in ((0, 0.5, 2, 2), (2, 1.0, 1, 2), (1, 0.1, 1, 4)):
        m = ris.ris_mask_generate(N, Hkv, mode, d, list(range(S)))
        assert ris.ris_attention_design(m, torch.bfloat16, D) == design
        base = ris.ris_attention_masked(m, q, k, v, rope=rope, out_dtype=torch.float32)
        out = ris.ris_attention_masked(m, q, k, big, rope=rope, out_dtype=torch.float32)
        torch.cuda.synchronize()
        ris.ris_device_status()
        m.free()
        assert torch.isfinite(out).all()
        scaled_back = out / (2.0 ** scale_exp)
        ref, _ = run_oracle(qn, kn, vn, mode, d, list(range(S)), 3, 1e6, 256)
        check_bf16_path(to_np(scaled_back), ref)
        # the same operands up to a power of two: within fp32 rounding of the unscaled output
        assert torch.allclose(scaled_back, base, rtol=1e-5, atol=1e-5)


# (N, mode, density, seeds, design, per_seed): the tiles, the register gather, the dense-suffix
# split, and the register gather's per-seed set loop
FP8_SCHEME_CASES = [(1200, 0, 0.5, [1, 2], 2, False), (1200, 0, 0.02, [1], 0, False), (3000, 1, 0.1, [1], 4, False),
                    (1300, 0, 0.03, [1, 2, 3], 0, True)]


@pytest.mark.parametrize("case", ["fp8", "both_large", "q_beyond_fp16"])
@pytest.mark.parametrize("N,mode,d,seeds,design,per_seed", FP8_SCHEME_CASES)
def test_fp8_score_scheme_and_its_fallback(N, mode, d, seeds, design, per_seed, case):
    """At head dim 128 with rotated bf16 inputs the tiles, the gather and the dense-suffix split
    take fp16 score products with e4m3 corrections when bounds of |q~| and |k~| allow (their
    product below about 1e5, each below 2^15 so that the fp16 hi parts stay finite); otherwise
    the call keeps the bf16 hi / lo scheme, chosen on the device. Queries and keys get one large
    channel each, in channel pairs where the other tensor is zero (so the scores stay moderate):
    at 9 they take the fp8 path; at 900 each the product rules it out; a query channel of 69632
    with keys scaled by 2^-7 passes the product rule but not fp16's range. Every case must match
    the oracle, every seed's output of a per-seed mask too."""
    Hq, Hkv, D = 6, 2, 128
    big_q, big_k, k_scale = {"fp8": (9.0, 9.0, 1.0), "both_large": (900.0, 900.0, 1.0),
                             "q_beyond_fp16": (69632.0, 1.0, 2.0 ** -7)}[case]
    (q, k, v), _ = make_inputs(N, Hq, Hkv, D, seed=67, outliers=True)
    q[:, :, 3] = big_q
    q[:, :, 5] = 0
    q[:, :, 5 + D // 2] = 0
    k.mul_(k_scale)
    k[:, :, 5] = big_k
    k[:, :, 3] = 0
    k[:, :, 3 + D // 2] = 0
    qn, kn, vn = to_np(q.cpu()), to_np(k.cpu()), to_np(v.cpu())
    m = ris.ris_mask_generate(N, Hkv, mode, d, seeds, per_seed=per_seed)
    assert ris.ris_attention_design(m, torch.bfloat16, D) == design
    out, lse = ris.ris_attention_masked(m, q, k, v, rope=ris.rope_cfg(3, 1e6, 256), out_dtype=torch.float32,
                                        return_lse=True)
    torch.cuda.synchronize()
    ris.ris_device_status()
    m.free()
    for s in range(len(seeds) if per_seed else 1):
        ref, ref_lse = run_oracle(qn, kn, vn, mode, d, seeds, 3, 1e6, 256, seed_index=s if per_seed else -1)
        check_bf16_path(to_np(out[s] if per_seed else out), ref)
        np.testing.assert_allclose(to_np(lse[s] if per_seed else lse).T, ref_lse, rtol=0, atol=2e-3)
