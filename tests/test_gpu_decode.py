"""GPU Hybrid Anchor decode vs the fp64 oracle: anchor keys bit-exact, rotated K cache, and the
decode step (one softmax over the frozen anchor merged with the sliding window)."""
import numpy as np
import pytest
import torch

import oracle as ora
from helpers import check_bf16_path, check_f32_path, make_inputs, oracle_rope, to_np
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def anchor_spec(N, mode, d, seeds, A=0, head_key=0, layer_key=0, sampler=0):
    return ora.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, n_anchor=A, head_key=head_key, layer_key=layer_key,
                        sampler=sampler)


@pytest.mark.parametrize("N,mode,d,S,A,sampler", [
    (1, 0, 0.05, 1, 0, 0), (33, 0, 0.3, 2, 0, 0), (300, 1, 0.05, 3, 2, 0), (1000, 0, 0.01, 10, 0, 0),
    (4133, 1, 0.013, 4, 5, 0), (700, 0, 0.05, 3, 0, 1), (900, 1, 0.05, 2, 1, 1), (500, 2, 0.01, 1, 0, 0),
    (65536, 0, 0.01, 10, 0, 0), (65536, 1, 0.01, 10, 0, 0)])
def test_anchor_matches_oracle(N, mode, d, S, A, sampler):
    seeds = list(range(3, 3 + S))
    opts = ris.mask_opts(local_window=9, n_anchor=A, layer_key=2, sampler=sampler)
    an = ris.ris_decode_anchor(N, 2, mode, d, seeds, opts=opts)
    t0, hk, n, keys, off = an.info()
    ref = ora.decode_anchor(anchor_spec(N, mode, d, seeds, A=A, layer_key=2, sampler=sampler))
    assert t0 == N and hk == 1 and n == ref.shape[0]
    np.testing.assert_array_equal(keys.cpu().numpy(), ref)
    np.testing.assert_array_equal(off.cpu().numpy(), [0, n])
    an.free()


def test_anchor_per_head():
    N, seeds, Hkv = 2000, [1, 2, 3], 4
    an = ris.ris_decode_anchor(N, Hkv, 0, 0.02, seeds, opts=ris.mask_opts(per_head=True))
    t0, hk, n, keys, off = an.info()
    keys, off = keys.cpu().numpy(), off.cpu().numpy()
    assert hk == Hkv
    for h in range(Hkv):
        ref = ora.decode_anchor(anchor_spec(N, 0, 0.02, seeds, head_key=h))
        np.testing.assert_array_equal(keys[off[h]:off[h + 1]], ref)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_rope_split_positions_and_parts(dtype):
    """Rotating a slice at pos0 equals that slice of the whole rotation, and hi (+ lo) matches
    the fp64 rotation to the precision of the split."""
    T, H, D, n_ctx = 3000, 2, 128, 4096
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 1024)
    (x, _, _), (xn, _, _) = make_inputs(T, H, 1, D, dtype=dtype, seed=9, outliers=True)
    hi, lo = ris.ris_rope_split(x, n_ctx, rope)
    hi2, lo2 = ris.ris_rope_split(x[1234:1300].contiguous(), n_ctx, rope, pos0=1234)
    torch.cuda.synchronize()
    assert torch.equal(hi[1234:1300], hi2)
    ref = ora.rope(xn, np.arange(T, dtype=np.float64), oracle_rope(3, 1e6, 1024), n_ctx)
    got = to_np(hi) + (to_np(lo) if lo is not None else 0.0)
    if dtype == torch.bfloat16:
        assert torch.equal(lo[1234:1300], lo2)
        assert np.abs(got - ref).max() <= 1e-5 * max(1.0, np.abs(ref).max())
    else:
        assert lo is None
        assert np.abs(got - ref).max() <= 4e-6 * max(1.0, np.abs(ref).max())


def _decode_case(N, T, Hq, Hkv, D, dtype, mode, d, seeds, steps, window, rope_kind=3, theta=1e6, native=256,
                 opts=None, split=True, out_dtype=None, seed=0, outliers=True):
    """Build the cache for positions 0..T-1, then decode each t in steps; compare with the oracle."""
    (q, k, v), (qn, kn, vn) = make_inputs(T, Hq, Hkv, D, dtype=dtype, seed=seed, outliers=outliers)
    rope = ris.rope_cfg(rope_kind, theta, native) if rope_kind else None
    k_hi, k_lo = ris.ris_rope_split(k, N, rope, split=split)
    an = ris.ris_decode_anchor(N, Hkv, mode, d, seeds, opts=opts)
    o = opts or ris.mask_opts()
    cfg = oracle_rope(rope_kind, theta, native)
    for t in steps:
        out, lse = ris.ris_decode_step(an, q[t].contiguous(), k_hi, k_lo, v, t, window, N, rope, out_dtype=out_dtype,
                                       return_lse=True)
        torch.cuda.synchronize()
        lists = []
        for g in range(Hkv) if o.per_head else [0]:
            spec = anchor_spec(N, mode, d, seeds, A=o.n_anchor, head_key=g if o.per_head else 0,
                               layer_key=o.layer_key, sampler=o.sampler)
            lists.append(ora.decode_anchor(spec))
        G = Hq // Hkv
        for g in range(Hkv):
            A = lists[g if o.per_head else 0]
            ref, ref_lse, _ = ora.decode_step(qn[t, g * G:(g + 1) * G], kn[:, g:g + 1], vn[:, g:g + 1], t, A, window,
                                              cfg, N)
            got = to_np(out[g * G:(g + 1) * G])
            if dtype == torch.float32:
                check_f32_path(got, ref)
                np.testing.assert_allclose(to_np(lse[g * G:(g + 1) * G]), ref_lse, rtol=1e-5, atol=1e-5)
            else:
                check_bf16_path(got, ref, out_bf16=(out_dtype == torch.bfloat16 or
                                                    (out_dtype is None and dtype == torch.bfloat16)))
                np.testing.assert_allclose(to_np(lse[g * G:(g + 1) * G]), ref_lse, rtol=0, atol=2e-3)
    an.free()


@pytest.mark.parametrize("mode,d,S,window,steps", [
    (0, 0.05, 3, 16, [300, 301, 333, 650]), (1, 0.05, 2, 1, [300, 302]), (0, 0.02, 5, 1000, [300, 420]),
    (2, 1.0, 1, 8, [300, 305])], ids=["stoch_w16", "struct_w1", "window_covers_all", "dense"])
def test_decode_small_bf16(mode, d, S, window, steps):
    _decode_case(300, 700, 12, 2, 128, torch.bfloat16, mode, d, list(range(S)), steps, window, out_dtype=torch.float32)


def test_decode_small_bf16_out_and_tinyllama_shape():
    _decode_case(500, 620, 32, 4, 64, torch.bfloat16, 1, 0.02, [7, 8], [500, 555, 619], 32, theta=1e4, native=64)


@pytest.mark.parametrize("Hq,Hkv,D", [(4, 4, 128), (6, 2, 64), (15, 3, 128)], ids=["mha_G1", "G3_d64", "G5"])
def test_decode_bf16_query_groups(Hq, Hkv, D):
    """Groups smaller than the 8 rows the score product carries (the other rows are zero)."""
    _decode_case(350, 420, Hq, Hkv, D, torch.bfloat16, 0, 0.05, [3, 4], [350, 377, 419], 24,
                 out_dtype=torch.float32)


def test_decode_fp32_path():
    _decode_case(257, 400, 4, 4, 64, torch.float32, 0, 0.1, [1], [257, 300, 399], 20, rope_kind=1, outliers=False)


def test_decode_per_head_and_draw_sampler():
    opts = ris.mask_opts(per_head=True, n_anchor=3, layer_key=5, sampler=ris.SAMPLER_DRAWS)
    _decode_case(800, 900, 6, 2, 128, torch.bfloat16, 0, 0.03, [2, 4], [800, 850, 899], 24, opts=opts,
                 out_dtype=torch.float32)


def test_decode_bf16_keys_without_low_part():
    """The cache may hold bf16 keys only (k_lo NULL): the bar still holds without outliers."""
    _decode_case(400, 500, 12, 2, 128, torch.bfloat16, 0, 0.05, [1, 2], [400, 470], 16, split=False,
                 out_dtype=torch.float32, outliers=False)


def test_decode_full_size_qwen_64k():
    """After the N=65536 prefill (Stochastic 1% x 10, YaRN s=2): the first generated tokens with
    the paper's 1024-token window."""
    N = 65536
    _decode_case(N, N + 8, 12, 2, 128, torch.bfloat16, 0, 0.01, list(range(10)), [N, N + 7], 1024, native=32768,
                 theta=1e6, out_dtype=torch.float32, seed=3)


def test_decode_rejects_bad_steps():
    (q, k, v), _ = make_inputs(200, 4, 2, 64, seed=1)
    an = ris.ris_decode_anchor(150, 2, 0, 0.05, [1])
    k_hi, k_lo = ris.ris_rope_split(k, 150, None)
    with pytest.raises(ris.RisError):
        ris.ris_decode_step(an, q[0].contiguous(), k_hi, k_lo, v, 149, 8, 150)  # before the first token
    with pytest.raises(ris.RisError):
        ris.ris_decode_step(an, q[0].contiguous(), k_hi, k_lo, v, 200, 8, 150)  # beyond the cache
    with pytest.raises(ris.RisError):
        ris.ris_decode_step(an, q[0].contiguous(), k_hi, k_lo, v, 160, 0, 150)  # empty window
    an.free()


def test_decode_device_position_and_graph_replay():
    """The position read from device memory, advanced by each step: one captured CUDA graph of
    the step replayed token after token gives the oracle's outputs for t0, t0 + 1, ..."""
    N, T, Hq, Hkv, D = 600, 700, 12, 2, 128
    (q, k, v), (qn, kn, vn) = make_inputs(T, Hq, Hkv, D, seed=21, outliers=True)
    rope = ris.rope_cfg(ris.ROPE_YARN, 1e6, 256)
    k_hi, k_lo = ris.ris_rope_split(k, N, rope)
    an = ris.ris_decode_anchor(N, Hkv, 1, 0.03, [5, 6])
    A = ora.decode_anchor(anchor_spec(N, 1, 0.03, [5, 6]))
    W = 48
    qbuf = torch.empty(Hq, D, dtype=q.dtype, device="cuda")
    out = torch.empty(Hq, D, dtype=torch.float32, device="cuda")
    t_dev = torch.tensor([N], dtype=torch.int64, device="cuda")
    qbuf.copy_(q[N])
    ris.ris_decode_step(an, qbuf, k_hi, k_lo, v, 0, W, N, rope, out=out, t_dev=t_dev, advance=True)  # allocates
    torch.cuda.synchronize()
    assert int(t_dev.item()) == N + 1
    ref, _, _ = ora.decode_step(qn[N], kn, vn, N, A, W, oracle_rope(3, 1e6, 256), N)
    check_bf16_path(to_np(out), ref)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        ris.ris_decode_step(an, qbuf, k_hi, k_lo, v, 0, W, N, rope, out=out, t_dev=t_dev, advance=True)
    for t in (N + 1, N + 2, N + 60):
        t_dev.fill_(t)
        qbuf.copy_(q[t])
        g.replay()
        torch.cuda.synchronize()
        assert int(t_dev.item()) == t + 1
        ref, _, _ = ora.decode_step(qn[t], kn, vn, t, A, W, oracle_rope(3, 1e6, 256), N)
        check_bf16_path(to_np(out), ref)
    ris.ris_device_status()
    # a device-side position past the cache is flagged and attends to nothing
    t_dev.fill_(T)
    g.replay()
    with pytest.raises(ris.RisError):
        ris.ris_device_status()
    ris.ris_device_status()  # the report cleared the flag
    an.free()


def test_decode_long_anchor_fold_beyond_shared_memory():
    """An anchor list long enough (about 42k keys, 167 cluster partials x 8 heads) that the
    final fold takes its fallback path (more partials than the shared memory holds)."""
    N = 65536
    _decode_case(N, N + 4, 16, 2, 64, torch.bfloat16, 0, 0.1, list(range(10)), [N, N + 3], 256, native=32768,
                 theta=1e6, out_dtype=torch.float32, seed=8)
