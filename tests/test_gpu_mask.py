"""GPU mask sampler vs the fp64 oracle: bitmap and CSR bit-exact (integer work)."""
import numpy as np
import pytest
import torch

import oracle as ora
from helpers import row_word_offset, sample_rows
from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def gpu_mask(N, mode, d, seeds, kv_heads=1, per_seed=False, W=1, A=0, per_head=False, layer_key=0, sampler=0):
    opts = ris.mask_opts(local_window=W, n_anchor=A, per_head=per_head, layer_key=layer_key, sampler=sampler)
    return ris.ris_mask_generate(N, kv_heads, mode, d, seeds, opts=opts, per_seed=per_seed)


def oracle_spec(N, mode, d, seeds, seed_index=-1, W=1, A=0, head_key=0, layer_key=0, sampler=0):
    return ora.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, seed_index=seed_index, local_window=W,
                        n_anchor=A, head_key=head_key, layer_key=layer_key, sampler=sampler)


def check_rows(m, specs, rows, check_bits=True):
    """specs[mask_id] is the oracle spec of that mask; compare the given rows."""
    d = m.info()
    N = d.N
    row_ptr = m.row_ptr().cpu().numpy()
    cols = m.cols().cpu().numpy()
    bitmap = m.bitmap().cpu().numpy().view(np.uint32) if check_bits else None
    assert row_ptr[0] == 0 and np.all(np.diff(row_ptr) >= 1)
    assert row_ptr[-1] == d.n_pairs == cols.shape[0]
    for mid, spec in enumerate(specs):
        off, ref = ora.mask_cols(spec, rows)
        for r, i in enumerate(rows):
            a, b = row_ptr[mid * N + i], row_ptr[mid * N + i + 1]
            np.testing.assert_array_equal(cols[a:b], ref[off[r]:off[r + 1]], err_msg=f"mask {mid} row {i}")
        if check_bits:
            words = ora.mask_bits(spec, rows)
            for r, i in enumerate(rows):
                nw = (i >> 5) + 1
                start = mid * d.words_per_mask + row_word_offset(int(i))
                np.testing.assert_array_equal(bitmap[start:start + nw], words[r, :nw],
                                              err_msg=f"bitmap mask {mid} row {i}")


@pytest.mark.parametrize("N,mode,d,S,W,A", [
    (1, 0, 0.05, 1, 1, 0), (33, 0, 0.3, 2, 1, 0), (100, 1, 0.05, 3, 1, 0), (257, 0, 0.01, 70, 1, 0),
    (300, 1, 0.2, 1, 4, 3), (513, 0, 1.0, 1, 1, 0), (700, 2, 0.01, 2, 1, 0), (1000, 1, 0.013, 10, 1, 0),
    (2048, 0, 0.05, 1, 1, 0)])
def test_mask_full_small(N, mode, d, S, W, A):
    seeds = list(range(100, 100 + S))
    m = gpu_mask(N, mode, d, seeds, W=W, A=A)
    if m.info().dense:
        assert m.info().n_pairs == N * (N + 1) // 2
        return
    check_rows(m, [oracle_spec(N, mode, d, seeds, W=W, A=A)], np.arange(N))


def test_mask_per_seed_and_per_head():
    N, seeds, Hkv = 400, [5, 6, 7], 2
    m = gpu_mask(N, 0, 0.05, seeds, kv_heads=Hkv, per_seed=True, per_head=True, layer_key=9)
    d = m.info()
    assert d.n_masks == 6 and d.heads_keyed == 2
    specs = [oracle_spec(N, 0, 0.05, seeds, seed_index=s, head_key=h, layer_key=9)
             for s in range(3) for h in range(Hkv)]
    check_rows(m, specs, np.arange(N))
    m2 = gpu_mask(N, 1, 0.05, seeds, per_seed=True)
    check_rows(m2, [oracle_spec(N, 1, 0.05, seeds, seed_index=s) for s in range(3)], np.arange(N))


# The five workload shapes: N, mode, density, seeds.
CONFIG_MASKS = [
    ("C1", 2048, 0, 0.05, 1), ("C2", 8192, 0, 0.01, 10), ("C3", 16384, 1, 0.01, 10),
    ("C4a", 32768, 0, 0.01, 70), ("C4b", 32768, 0, 0.05, 10), ("C5s", 65536, 0, 0.01, 10),
    ("C5t", 65536, 1, 0.01, 10),
]


@pytest.mark.parametrize("name,N,mode,d,S", CONFIG_MASKS, ids=[c[0] for c in CONFIG_MASKS])
def test_mask_config_sizes_sampled_rows(name, N, mode, d, S):
    seeds = list(range(S))
    m = gpu_mask(N, mode, d, seeds)
    rows = sample_rows(N, 48, seed=N)
    check_rows(m, [oracle_spec(N, mode, d, seeds)], rows)
    # pair count matches its expectation within binomial bounds (property at any size)
    info = m.info()
    if mode == 0:
        U = 1 - (1 - d) ** S
        T = N * (N - 1) / 2
        assert abs(info.n_pairs - N - U * T) < 6 * np.sqrt(T * U * (1 - U))
    m.free()
    torch.cuda.synchronize()


def test_mask_u32_columns_beyond_65536():
    """N > 65536 switches the key lists to 32-bit indices."""
    N = 65600
    m = gpu_mask(N, 0, 0.0005, [1])
    assert m.info().col_bytes == 4
    check_rows(m, [oracle_spec(N, 0, 0.0005, [1])], sample_rows(N, 8, seed=3), check_bits=False)


def test_mask_deterministic_and_keyed():
    a = gpu_mask(500, 0, 0.1, [3]).cols().cpu()
    b = gpu_mask(500, 0, 0.1, [3]).cols().cpu()
    assert torch.equal(a, b)
    c = gpu_mask(500, 0, 0.1, [3], layer_key=1).cols().cpu()
    assert a.shape != c.shape or not torch.equal(a, c)


# ----------------------------------------------------------------------------- index-draw sampler
@pytest.mark.parametrize("N,mode,d,S,W,A", [
    (1, 0, 0.05, 1, 1, 0), (2, 0, 0.9, 3, 1, 0), (33, 0, 0.3, 2, 1, 0), (100, 1, 0.05, 3, 1, 0),
    (300, 1, 0.2, 1, 4, 3), (513, 0, 1.0, 1, 1, 0), (1000, 1, 0.013, 10, 1, 0), (2048, 0, 0.05, 7, 1, 0),
    (4133, 0, 0.002, 1, 1, 0), (3000, 0, 0.0001, 2, 5, 0)])
def test_draw_sampler_full_small(N, mode, d, S, W, A):
    """Index draws (with replacement, causal filter, merged) bit-exact against the oracle,
    including K = 0 draws (forced set only) and density 1 (dense)."""
    seeds = list(range(40, 40 + S))
    m = gpu_mask(N, mode, d, seeds, W=W, A=A, sampler=1)
    if m.info().dense:
        assert m.info().n_pairs == N * (N + 1) // 2
        return
    assert m.info().params.draws == ris.ris_resolve_params(N, mode, d)["draws"]
    check_rows(m, [oracle_spec(N, mode, d, seeds, W=W, A=A, sampler=1)], np.arange(N))


def test_draw_sampler_per_seed_and_per_head():
    N, seeds, Hkv = 600, [5, 6, 7], 2
    m = gpu_mask(N, 0, 0.05, seeds, kv_heads=Hkv, per_seed=True, per_head=True, layer_key=9, sampler=1)
    specs = [oracle_spec(N, 0, 0.05, seeds, seed_index=s, head_key=h, layer_key=9, sampler=1)
             for s in range(3) for h in range(Hkv)]
    check_rows(m, specs, np.arange(N))
    m2 = gpu_mask(N, 1, 0.05, seeds, per_seed=True, sampler=1)
    check_rows(m2, [oracle_spec(N, 1, 0.05, seeds, seed_index=s, sampler=1) for s in range(3)], np.arange(N))


@pytest.mark.parametrize("N,mode,d,S", [(65536, 0, 0.01, 10), (65536, 1, 0.01, 10), (32768, 0, 0.01, 70)])
def test_draw_sampler_config_sizes_sampled_rows(N, mode, d, S):
    seeds = list(range(S))
    m = gpu_mask(N, mode, d, seeds, sampler=1)
    check_rows(m, [oracle_spec(N, mode, d, seeds, sampler=1)], sample_rows(N, 48, seed=N + mode))


# ----------------------------------------------------------------------------- paper geometry and sweep
@pytest.mark.parametrize("mode", [0, 1])
def test_mask_paper_geometry_full_size(mode):
    """Local window 1024 + 4 anchors at N=65536 (both modes, 1% x 10): sampled rows bit-exact,
    every row keeps its whole window and the anchors."""
    N, seeds = 65536, list(range(10))
    m = gpu_mask(N, mode, 0.01, seeds, W=ris.PRESET_LOCAL_WINDOW, A=ris.PRESET_ANCHORS)
    rows = sample_rows(N, 32, seed=77 + mode)
    check_rows(m, [oracle_spec(N, mode, 0.01, seeds, W=1024, A=4)], rows)
    counts = np.diff(m.row_ptr().cpu().numpy())
    i = np.arange(N)
    assert (counts >= np.minimum(i + 1, 1024)).all()
    assert (counts[1027:] >= 1024 + 4).all()  # window and anchors are disjoint from row 1027 on


@pytest.mark.parametrize("d,S", [(0.001, 200), (0.003, 150), (0.005, 100), (0.009, 50)])
def test_mask_sub1pct_structural_sweep(d, S):
    """Sub-1% Structural sweep points at N=65536: B_max as the paper's table, sampled rows bit-exact."""
    N, seeds = 65536, list(range(S))
    m = gpu_mask(N, 1, d, seeds)
    p = m.info().params
    assert p.bmax == int(np.floor(d * N + 0.5)) and p.block == min(N // 10, p.bmax)
    check_rows(m, [oracle_spec(N, 1, d, seeds)], sample_rows(N, 16, seed=int(d * 1e4) + S))


@pytest.mark.parametrize("N,mode,d,S,W,per_head", [
    (3000, 1, 0.1, 2, 1, False), (4100, 1, 0.08, 1, 40, False), (3300, 1, 0.1, 1, 700, True),
    (2900, 0, 0.01, 3, 300, False), (1500, 1, 0.002, 1, 600, False), (2000, 1, 0.05, 1, 1, False),
    (700, 0, 0.02, 1, 900, False)])
def test_dense_suffix_is_the_tail_of_every_row(N, mode, d, S, W, per_head):
    """The dense-suffix split's premise on real masks: every key from lo(i) (the earlier of the
    row's Structural block start, for blocks of >= 256 tokens, and its local window start,
    for windows of >= 256) up to i is kept, so those keys end the row's ascending list; and
    the mask description's suffix pair count is the brute-force sum of their lengths."""
    m = gpu_mask(N, mode, d, list(range(S)), kv_heads=2, W=W, per_head=per_head)
    info = m.info()
    block = info.params.block if (mode == 1 and info.params.block >= 256) else 0
    allowed = block > 0 or W >= 256

    def lo(i):
        v = i
        if block:
            v = min(v, (i // block) * block)
        if W > 1:
            v = min(v, max(0, i - W + 1))
        return v

    expect = sum(i - lo(i) + 1 for i in range(N)) if allowed else 0
    assert info.suffix_pairs == expect
    if allowed:
        row_ptr = m.row_ptr().cpu().numpy()
        cols = m.cols().cpu().numpy().astype(np.int64)
        for mid in range(info.n_masks):
            for i in range(N):
                a, b = row_ptr[mid * N + i], row_ptr[mid * N + i + 1]
                tail = i - lo(i) + 1
                assert b - a >= tail
                np.testing.assert_array_equal(cols[b - tail:b], np.arange(lo(i), i + 1), err_msg=f"row {i}")
    m.free()
