"""Pins of the fp64 oracle against facts outside itself (no GPU).

Every test here checks the oracle against something it does not compute: values the paper
prints (tests/golden), an independent library implementation (the Triton interpreter's
Philox4x32-10, torch's fp64 scaled-dot-product attention), closed forms, invariants and
brute force on tiny inputs. A plausible slip in the oracle -- a dropped term, a wrong sign
or index, a transposed operand -- fails at least one of them.
"""
import math
import os
import subprocess
import sys
import textwrap

import numpy as np
import pytest
import torch

from conftest import ROOT, golden

pytestmark = pytest.mark.filterwarnings("ignore::DeprecationWarning")


# ----------------------------------------------------------------------------- Philox
_TRITON_PHILOX = textwrap.dedent(
    """
    import os, sys
    os.environ["TRITON_INTERPRET"] = "1"
    import numpy as np, torch, triton, triton.language as tl

    @triton.jit
    def k(c0p, c1p, c2p, c3p, k0p, k1p, o0, o1, o2, o3, n: tl.constexpr):
        offs = tl.arange(0, n)
        u = tl.uint32
        c0 = tl.load(c0p + offs).to(u, bitcast=True)
        c1 = tl.load(c1p + offs).to(u, bitcast=True)
        c2 = tl.load(c2p + offs).to(u, bitcast=True)
        c3 = tl.load(c3p + offs).to(u, bitcast=True)
        k0 = tl.load(k0p + offs).to(u, bitcast=True)
        k1 = tl.load(k1p + offs).to(u, bitcast=True)
        a, b, c, d = tl.philox_impl(c0, c1, c2, c3, k0, k1, 10)
        tl.store(o0 + offs, a.to(tl.int32, bitcast=True))
        tl.store(o1 + offs, b.to(tl.int32, bitcast=True))
        tl.store(o2 + offs, c.to(tl.int32, bitcast=True))
        tl.store(o3 + offs, d.to(tl.int32, bitcast=True))

    data = np.load(sys.argv[1])
    ctr, key = data["ctr"].view(np.int32), data["key"].view(np.int32)
    n = ctr.shape[0]
    ins = [torch.from_numpy(np.ascontiguousarray(ctr[:, i])) for i in range(4)]
    ins += [torch.from_numpy(np.ascontiguousarray(key[:, i])) for i in range(2)]
    outs = [torch.empty(n, dtype=torch.int32) for _ in range(4)]
    k[(1,)](*ins, *outs, n=n)
    np.save(sys.argv[2], np.stack([o.numpy() for o in outs], 1).view(np.uint32))
    """
)


def test_philox_matches_triton_interpreter(oracle, tmp_path):
    """Philox4x32-10 equals the independent implementation in Triton's random module, run on
    the CPU by Triton's interpreter (Salmon et al. SC'11 constants, 10 rounds)."""
    pytest.importorskip("triton")
    rng = np.random.default_rng(1234)
    n = 256
    ctr = rng.integers(0, 2**32, size=(n, 4), dtype=np.uint64).astype(np.uint32)
    key = rng.integers(0, 2**32, size=(n, 2), dtype=np.uint64).astype(np.uint32)
    ctr[:4] = 0  # the all-zero counter with a few keys
    key[0] = 0
    inp, outp, script = tmp_path / "in.npz", tmp_path / "out.npy", tmp_path / "tp.py"
    np.savez(inp, ctr=ctr, key=key)
    script.write_text(_TRITON_PHILOX)
    env = dict(os.environ, TRITON_INTERPRET="1")
    subprocess.run([sys.executable, str(script), str(inp), str(outp)], check=True, env=env,
                   timeout=300)
    ref = np.load(outp)
    got = oracle.philox(ctr, key)
    np.testing.assert_array_equal(got, ref)


def test_philox_words_uniform(oracle):
    """Philox words are uniform on [0, 2^32): chi-square over 64 buckets and mean."""
    n = 1 << 16
    ctr = np.zeros((n, 4), np.uint32)
    ctr[:, 0] = np.arange(n)
    ctr[:, 1] = 7
    key = np.tile(np.array([[5, 9]], np.uint32), (n, 1))
    w = oracle.philox(ctr, key).ravel().astype(np.float64)
    hist = np.bincount((w // 2**26).astype(np.int64), minlength=64)
    e = w.size / 64
    chi2 = ((hist - e) ** 2 / e).sum()
    assert chi2 < 63 + 6 * math.sqrt(2 * 63)
    assert abs(w.mean() / 2**32 - 0.5) < 5 * math.sqrt(1 / 12 / w.size)


# ----------------------------------------------------------------------------- thresholds
def test_threshold_closed_form(oracle):
    assert oracle.threshold(0.0) == 0
    assert oracle.threshold(1.0) == 2**32
    assert oracle.threshold(0.5) == 2**31
    assert oracle.threshold(0.25) == 2**30
    assert oracle.threshold(2.0**-32) == 1
    assert oracle.threshold(1.0 - 2.0**-33) == 2**32  # rounds up to "always"


@pytest.mark.parametrize("p", [0.01, 0.05, 0.3])
def test_threshold_gives_bernoulli_p(oracle, p):
    """The fraction of Philox words below thr(p) is p within 5 sigma."""
    n = 1 << 17
    ctr = np.zeros((n, 4), np.uint32)
    ctr[:, 0] = np.arange(n)
    key = np.tile(np.array([[11, 0]], np.uint32), (n, 1))
    w = oracle.philox(ctr, key).ravel().astype(np.uint64)
    frac = (w < oracle.threshold(p)).mean()
    assert abs(frac - p) < 5 * math.sqrt(p * (1 - p) / w.size)


# ----------------------------------------------------------------------------- Structural geometry
def test_bmax_matches_paper_table(oracle):
    """B_max = round(d N) reproduces the B_max column of the sub-1% sweet-spot table."""
    rows = golden("bmax_table.txt")
    assert len(rows) == 10
    for N, dpct, bmax in rows:
        g = oracle.structural(int(N), float(dpct) / 100.0)
        assert g["K"] == int(bmax), (dpct, g)
        # B = min(0.1 N, B_max): at N = 65536 the tenth (6553) never binds
        assert g["B"] == int(bmax)


def _brute_clique(N, B):
    i = np.arange(N)[:, None]
    j = np.arange(N)[None, :]
    return (j <= i) & (i // B == j // B)


@pytest.mark.parametrize("N,d", [(10, 0.05), (37, 0.2), (100, 0.05), (1000, 0.01), (999, 0.013),
                                 (16384, 0.01)])
def test_clique_count_bruteforce(oracle, N, d):
    g = oracle.structural(N, d)
    B = g["B"]
    assert B == max(1, min(N // 10, int(math.floor(d * N + 0.5))))
    if N <= 1000:
        assert _brute_clique(N, B).sum() == g["C"]
    else:  # count per block: full blocks of B, one partial block
        sizes = [min(B, N - s) for s in range(0, N, B)]
        assert sum(s * (s + 1) // 2 for s in sizes) == g["C"]
    assert g["d_clique"] == pytest.approx(g["C"] / N**2, rel=1e-15)
    assert g["d_global"] == pytest.approx(max(0.0, d - g["C"] / N**2), abs=1e-18)


def test_structural_mask_cliques_and_global(oracle):
    """Structural mask = causal cliques (always kept) + global draws of density d_global."""
    N, d, S = 600, 0.05, 4
    spec = oracle.MaskSpec(N=N, mode=oracle.MODE_STRUCTURAL, density=d, seeds=[3, 4, 5, 6])
    m = oracle.mask_dense(spec)
    g = oracle.structural(N, d)
    cl = _brute_clique(N, g["B"])
    assert m[cl].all()
    assert not np.triu(m, 1).any()
    off = np.tril(np.ones((N, N), bool), -1) & ~cl
    p = 1 - (1 - g["d_global"]) ** S
    frac = m[off].mean()
    assert abs(frac - p) < 5 * math.sqrt(p * (1 - p) / off.sum())


# ----------------------------------------------------------------------------- Stochastic masks
def test_union_coverage_paper_values(oracle):
    """U = 1 - (1-d)^N reproduces the paper's 50.5% and 97.2% (to the printed decimal)."""
    for d, n, upct in golden("union_coverage.txt"):
        U = oracle.union_coverage(float(d), int(n))
        assert abs(100 * U - float(upct)) <= 0.05 + 1e-9


@pytest.mark.parametrize("d,S", [(0.01, 70), (0.05, 70), (0.05, 1)])
def test_union_mask_density_matches_coverage(oracle, d, S):
    """The master mask's off-diagonal density is U = 1-(1-d)^S within 5 sigma: every seed is
    OR-merged (Eq. union_coverage; Methods, Memory-Bounded Geometry Generation)."""
    N = 400
    spec = oracle.MaskSpec(N=N, mode=oracle.MODE_STOCHASTIC, density=d, seeds=list(range(S)))
    m = oracle.mask_dense(spec)
    low = np.tril(np.ones((N, N), bool), -1)
    U = oracle.union_coverage(d, S)
    frac = m[low].mean()
    assert abs(frac - U) < 5 * math.sqrt(U * (1 - U) / low.sum())
    assert np.diag(m).all() and not np.triu(m, 1).any()


def test_union_is_or_of_per_seed_masks(oracle):
    N, seeds = 300, [10, 20, 30]
    for mode in (oracle.MODE_STOCHASTIC, oracle.MODE_STRUCTURAL):
        u = oracle.mask_dense(oracle.MaskSpec(N=N, mode=mode, density=0.04, seeds=seeds))
        per = [oracle.mask_dense(oracle.MaskSpec(N=N, mode=mode, density=0.04, seeds=seeds,
                                                 seed_index=s)) for s in range(3)]
        np.testing.assert_array_equal(u, per[0] | per[1] | per[2])
        assert not (per[0] == per[1]).all()


def test_row_counts_binomial(oracle):
    """Per-row off-diagonal counts of one seed follow Binomial(i, d): total within 5 sigma and
    the per-row spread matches the binomial variance."""
    N, d = 2048, 0.05
    spec = oracle.MaskSpec(N=N, mode=oracle.MODE_STOCHASTIC, density=d, seeds=[0])
    c = oracle.mask_counts(spec) - 1  # diagonal is forced
    i = np.arange(N)
    n = i.sum()
    assert abs(c.sum() - d * n) < 5 * math.sqrt(n * d * (1 - d))
    z = (c - d * i)[1:] / np.sqrt(i[1:] * d * (1 - d))
    assert abs(z.mean()) < 5 / math.sqrt(N) and 0.8 < z.std() < 1.2


def test_columns_uniform(oracle):
    """Stochastic Mode samples keys uniformly: keep rate per key column bucket is flat (chi2)."""
    N, d = 1024, 0.1
    m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=oracle.MODE_STOCHASTIC, density=d, seeds=[2]))
    low = np.tril(np.ones((N, N), bool), -1)
    kept = (m & low).sum(0)
    trials = low.sum(0)
    b = 16
    kb = kept.reshape(b, -1).sum(1)
    tb = trials.reshape(b, -1).sum(1)
    chi2 = (((kb - d * tb) ** 2) / (d * (1 - d) * tb)).sum()
    assert chi2 < b + 6 * math.sqrt(2 * b)


def test_density_one_is_dense_causal(oracle):
    N = 130
    tri = np.tril(np.ones((N, N), bool))
    for mode in (0, 1, 2):
        m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=mode, density=1.0, seeds=[0]))
        np.testing.assert_array_equal(m, tri)
    m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=oracle.MODE_DENSE, density=0.01, seeds=[0]))
    np.testing.assert_array_equal(m, tri)


def test_forced_window_and_anchors(oracle):
    N, W, A = 300, 5, 3
    m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=0, density=0.001, seeds=[1], local_window=W,
                                          n_anchor=A))
    for i in range(N):
        for j in range(max(0, i - W + 1), i + 1):
            assert m[i, j]
        for j in range(min(A, i + 1)):
            assert m[i, j]
    assert not np.triu(m, 1).any()


def test_keys_change_the_draw(oracle):
    base = dict(N=256, mode=0, density=0.1, seeds=[7])
    m0 = oracle.mask_dense(oracle.MaskSpec(**base))
    np.testing.assert_array_equal(m0, oracle.mask_dense(oracle.MaskSpec(**base)))
    assert (m0 != oracle.mask_dense(oracle.MaskSpec(**base, head_key=1))).any()
    assert (m0 != oracle.mask_dense(oracle.MaskSpec(**base, layer_key=1))).any()
    assert (m0 != oracle.mask_dense(oracle.MaskSpec(**dict(base, seeds=[8])))).any()


def test_bits_and_cols_agree(oracle):
    spec = oracle.MaskSpec(N=200, mode=1, density=0.07, seeds=[1, 2])
    bits = oracle.mask_bits(spec)
    off, cols = oracle.mask_cols(spec)
    for i in range(200):
        js = cols[off[i]:off[i + 1]]
        b = np.zeros(bits.shape[1] * 32, bool)
        b[js] = True
        words = np.packbits(b.reshape(-1, 32)[:, ::-1], axis=1, bitorder="big").view(">u4").ravel()
        np.testing.assert_array_equal(words.astype(np.uint32), bits[i])


# ----------------------------------------------------------------------------- RoPE
def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def test_rope_plain_equals_complex_rotation(oracle):
    """Rotate-half RoPE is the complex product (x_c + i x_{c+D/2}) e^{i p f_c}, f_c = theta^(-2c/D)."""
    N, H, D, theta = 50, 3, 64, 1e4
    x = _rand((N, H, D), 0)
    pos = np.arange(N, dtype=np.float64)
    got = oracle.rope(x, pos, oracle.RopeCfg(kind=oracle.ROPE_PLAIN, theta=theta, native_len=4096), N)
    f = theta ** (-np.arange(0, D, 2, dtype=np.float64) / D)
    z = (x[..., : D // 2] + 1j * x[..., D // 2:]) * np.exp(1j * pos[:, None, None] * f)
    np.testing.assert_allclose(got, np.concatenate([z.real, z.imag], -1), rtol=0, atol=1e-12)


@pytest.mark.parametrize("kind", [2, 3])
def test_rope_factor_one_equals_plain(oracle, kind):
    """Inside the native window the factor is 1 and every method equals plain RoPE."""
    N, H, D = 64, 2, 128
    x = _rand((N, H, D), 1)
    pos = np.arange(N, dtype=np.float64)
    plain = oracle.rope(x, pos, oracle.RopeCfg(kind=1, native_len=128), N)
    ext = oracle.rope(x, pos, oracle.RopeCfg(kind=kind, native_len=128), N)
    np.testing.assert_allclose(ext, plain, rtol=0, atol=1e-13)


def test_rope_linear_compresses_positions(oracle):
    """Linear interpolation at position p equals plain RoPE at position p / s."""
    N, H, D, L = 256, 2, 64, 64
    cfg = oracle.RopeCfg(kind=2, theta=1e4, native_len=L)
    s = oracle.resolve_factor(cfg, N)
    assert s == 4.0
    x = _rand((N, H, D), 2)
    pos = np.arange(N, dtype=np.float64)
    a = oracle.rope(x, pos, cfg, N)
    b = oracle.rope(x, pos / s, oracle.RopeCfg(kind=1, theta=1e4, native_len=L), N)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)


def test_yarn_frequency_bands_and_mscale(oracle):
    """YaRN: wavelengths much shorter than the native window keep their frequency (r > beta),
    those longer than it are interpolated by s (r < alpha), the temperature factor is
    0.1 ln s + 1 (Peng et al. 2023), and the interpolated band lies between the two."""
    D, theta, L, N = 128, 1e6, 32768, 65536
    cfg = oracle.RopeCfg(kind=3, theta=theta, native_len=L)
    f, ms = oracle.rope_freqs(cfg, N, D)
    plain, _ = oracle.rope_freqs(oracle.RopeCfg(kind=1, theta=theta, native_len=L), N, D)
    s = 2.0
    wavelength = 2 * np.pi / plain
    r = L / wavelength
    hi, lo = r > 32, r < 1
    assert hi.any() and lo.any() and (~hi & ~lo).any()
    np.testing.assert_allclose(f[hi], plain[hi], rtol=1e-15)
    np.testing.assert_allclose(f[lo], plain[lo] / s, rtol=1e-15)
    mid = ~hi & ~lo
    assert np.all(f[mid] <= plain[mid]) and np.all(f[mid] >= plain[mid] / s)
    assert ms == pytest.approx(1.0 + 0.1 * math.log(2.0), rel=1e-15)


def test_yarn_mid_band_hand_worked(oracle):
    """A frequency inside YaRN's ramp, worked by hand from Peng et al. 2023 (NTK-by-parts,
    alpha = 1, beta = 32): head dim 8, base 1e4, native window L = 64, N = 256 (s = 4).
    Pair 0 has base frequency 1, wavelength 2 pi, so r = 64 / (2 pi) = 10.18591636 rotations per
    window; the ramp gives gamma = (r - 1) / 31 = 0.29631988 and the frequency
    (1 - gamma) * 1/4 + gamma * 1 = 0.47223991. Pair 1 (base 0.1, r = 1.01859164) sits just
    inside the ramp: gamma = 0.00059973, frequency 0.02504498. The temperature is
    0.1 ln 4 + 1 = 1.13862944. A unit vector rotated at position p turns by p times the
    frequency and is scaled by the temperature."""
    D, N = 8, 256
    cfg = oracle.RopeCfg(kind=3, theta=1e4, native_len=64)
    hand_f = {0: 0.47223991188, 1: 0.02504497976}
    hand_ms = 1.13862943611
    for c, f in hand_f.items():
        x = np.zeros((2, 1, D))
        x[:, 0, c] = 1.0
        y = oracle.rope(x, [1.0, 3.0], cfg, N)
        for row, p in enumerate((1.0, 3.0)):
            a, b = y[row, 0, c], y[row, 0, c + D // 2]
            assert math.hypot(a, b) == pytest.approx(hand_ms, abs=1e-10)
            assert math.atan2(b, a) == pytest.approx(p * f, abs=1e-10)


@pytest.mark.parametrize("kind", [1, 2, 3])
def test_rope_norm_and_relative_position(oracle, kind):
    """Each rotated pair keeps its norm (times mscale), and <R(p)q, R(p')k> depends on p - p' only."""
    N, H, D, L = 512, 1, 64, 128
    cfg = oracle.RopeCfg(kind=kind, theta=1e4, native_len=L)
    _, ms = oracle.rope_freqs(cfg, N, D)
    q = _rand((1, H, D), 3)
    k = _rand((1, H, D), 4)
    qa = oracle.rope(q, [100.0], cfg, N)
    pair = lambda t: np.hypot(t[..., : D // 2], t[..., D // 2:])
    np.testing.assert_allclose(pair(qa), ms * pair(q), rtol=1e-12)
    dots = []
    for shift in (0.0, 37.0, 300.0):
        a = oracle.rope(q, [100.0 + shift], cfg, N)
        b = oracle.rope(k, [40.0 + shift], cfg, N)
        dots.append(float((a * b).sum()))
    np.testing.assert_allclose(dots, dots[0], rtol=1e-10)


# ----------------------------------------------------------------------------- attention
def _sdpa(q, k, v, mask, G):
    """torch fp64 SDPA with an explicit boolean mask; KV heads repeated G times (head h -> h // G)."""
    qt = torch.from_numpy(q).permute(1, 0, 2)
    kt = torch.from_numpy(k).permute(1, 0, 2).repeat_interleave(G, 0)
    vt = torch.from_numpy(v).permute(1, 0, 2).repeat_interleave(G, 0)
    m = torch.from_numpy(mask)
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=m)
    s = (qt @ kt.transpose(1, 2)) / math.sqrt(q.shape[-1])
    lse = torch.logsumexp(s.masked_fill(~m, float("-inf")), -1)
    return o.permute(1, 0, 2).numpy(), lse.permute(1, 0).numpy()


@pytest.mark.parametrize("mode,d,S,Hq,Hkv,D", [(0, 0.05, 3, 4, 2, 64), (1, 0.05, 2, 6, 2, 32),
                                              (0, 0.3, 1, 3, 1, 16), (2, 1.0, 1, 4, 4, 64)])
def test_attention_matches_sdpa_with_bool_mask(oracle, mode, d, S, Hq, Hkv, D):
    """Oracle attention = torch fp64 SDPA on the explicit boolean master mask, GQA head map h -> h // G."""
    N = 193
    spec = oracle.MaskSpec(N=N, mode=mode, density=d, seeds=list(range(S)))
    q, k, v = _rand((N, Hq, D), 5), _rand((N, Hkv, D), 6), _rand((N, Hkv, D), 7)
    out, lse, off, cols = oracle.sparse_attention(q, k, v, spec, None)
    ref, ref_lse = _sdpa(q, k, v, oracle.mask_dense(spec), Hq // Hkv)
    np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-12, atol=1e-12)


def test_density_one_equals_sdpa_causal(oracle):
    N, H, D = 150, 2, 32
    q, k, v = _rand((N, H, D), 8), _rand((N, H, D), 9), _rand((N, H, D), 10)
    out, _, _, _ = oracle.sparse_attention(q, k, v, oracle.MaskSpec(N=N, mode=0, density=1.0, seeds=[0]))
    ref = torch.nn.functional.scaled_dot_product_attention(
        *[torch.from_numpy(t).permute(1, 0, 2) for t in (q, k, v)], is_causal=True).permute(1, 0, 2)
    np.testing.assert_allclose(out, ref.numpy(), rtol=1e-10, atol=1e-12)


def test_attention_constant_values_and_single_key(oracle):
    """V = 1 gives 1 everywhere; a row whose key set is itself returns its own value row."""
    N, Hq, Hkv, D = 120, 4, 2, 16
    q, k = _rand((N, Hq, D), 11), _rand((N, Hkv, D), 12)
    spec = oracle.MaskSpec(N=N, mode=0, density=0.2, seeds=[4])
    out, _, _, _ = oracle.sparse_attention(q, k, np.ones((N, Hkv, D)), spec)
    np.testing.assert_allclose(out, 1.0, rtol=0, atol=1e-13)
    v = _rand((N, Hkv, D), 13)
    tiny = oracle.MaskSpec(N=N, mode=0, density=1e-12, seeds=[4])  # only the diagonal survives
    out, lse, off, cols = oracle.sparse_attention(q, k, v, tiny)
    np.testing.assert_array_equal(cols, np.arange(N))
    np.testing.assert_allclose(out, np.repeat(v, Hq // Hkv, axis=1), rtol=0, atol=1e-14)


def test_attention_with_rope_is_rope_then_attention(oracle):
    """The whole path rotates q at its own row positions and k at 0..N-1, then attends."""
    N, Hq, Hkv, D = 160, 4, 2, 32
    q, k, v = _rand((N, Hq, D), 14), _rand((N, Hkv, D), 15), _rand((N, Hkv, D), 16)
    cfg = oracle.RopeCfg(kind=3, theta=1e4, native_len=64)
    spec = oracle.MaskSpec(N=N, mode=0, density=0.1, seeds=[1, 2])
    rows = np.array([0, 5, 77, 159])
    out, lse, _, _ = oracle.sparse_attention(q, k, v, spec, cfg, rows=rows)
    pos = np.arange(N, dtype=np.float64)
    qr, kr = oracle.rope(q, pos, cfg, N), oracle.rope(k, pos, cfg, N)
    ref, ref_lse = _sdpa(qr, kr, v, oracle.mask_dense(spec), Hq // Hkv)
    np.testing.assert_allclose(out, ref[rows], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse[rows], rtol=1e-12, atol=1e-12)


# ----------------------------------------------------------------------------- index-draw sampler
def _triton_philox(tmp_path, ctr, key):
    n = len(ctr)
    n2 = 1 << max(0, (n - 1).bit_length())  # the kernel's arange needs a power of two
    ctr = np.concatenate([ctr, np.zeros((n2 - n, 4), np.uint32)])
    key = np.concatenate([key, np.zeros((n2 - n, 2), np.uint32)])
    inp, outp, script = tmp_path / "din.npz", tmp_path / "dout.npy", tmp_path / "dtp.py"
    np.savez(inp, ctr=ctr, key=key)
    script.write_text(_TRITON_PHILOX)
    env = dict(os.environ, TRITON_INTERPRET="1")
    subprocess.run([sys.executable, str(script), str(inp), str(outp)], check=True, env=env, timeout=300)
    return np.load(outp)[:n]


def test_draw_sampler_matches_triton_draws(oracle, tmp_path):
    """Index-draw sampler (the torch.randint wording of Methods, Memory-Bounded Geometry
    Generation): the rows' key sets are rebuilt here from draws made by Triton's independent
    Philox (counter (t/4, i, stream+2, layer_key), key (seed, head_key), word t mod 4), mapped
    to j = floor(u N / 2^32), causally filtered and merged, plus the forced diagonal and, for
    Structural, the block clique."""
    pytest.importorskip("triton")
    N, seeds = 500, [3, 9]
    rows = np.array([0, 1, 37, 250, 499], dtype=np.int64)
    cases = [(oracle.MODE_STOCHASTIC, 0.04, 0, 0), (oracle.MODE_STRUCTURAL, 0.06, 2, 5)]
    ctr, key, meta = [], [], []
    for mode, d, hk, lk in cases:
        if mode == oracle.MODE_STRUCTURAL:
            g = oracle.structural(N, d)
            K, stream = int(math.floor(g["d_global"] * N + 0.5)), 3
        else:
            K, stream = int(math.floor(d * N + 0.5)), 2
        assert K > 0
        for i in rows:
            for s in seeds:
                for t in range(K):
                    ctr.append((t // 4, i, stream, lk))
                    key.append((s, hk))
                    meta.append((0, mode, int(i), t % 4))
    ctr = np.array(ctr, dtype=np.uint32)
    key = np.array(key, dtype=np.uint32)
    words = _triton_philox(tmp_path, ctr, key)
    u = words[np.arange(len(meta)), [m[3] for m in meta]].astype(np.uint64)
    j = (u * np.uint64(N)) >> np.uint64(32)
    for mode, d, hk, lk in cases:
        spec = oracle.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, head_key=hk, layer_key=lk, sampler=1)
        off, cols = oracle.mask_cols(spec, rows)
        B = oracle.structural(N, d)["B"] if mode == oracle.MODE_STRUCTURAL else None
        for r, i in enumerate(rows):
            sel = np.array([m[1] == mode and m[2] == i for m in meta])
            want = {int(x) for x in j[sel] if x < i} | {int(i)}
            if B is not None:
                want |= set(range((i // B) * B, i + 1))
            assert set(cols[off[r]:off[r + 1]].tolist()) == want, (mode, i)
            assert (np.diff(cols[off[r]:off[r + 1]]) > 0).all()


def test_draw_sampler_density(oracle):
    """S seeds of K = round(dN) draws over [0, N): each earlier key of row i is hit with
    probability q = 1 - (1 - 1/N)^(S K); the total kept count is within 5 sigma of q * sum(i)."""
    N, d, S = 1000, 0.02, 5
    spec = oracle.MaskSpec(N=N, mode=0, density=d, seeds=list(range(S)), sampler=1)
    c = oracle.mask_counts(spec) - 1  # diagonal forced
    K = int(math.floor(d * N + 0.5))
    q = 1 - (1 - 1 / N) ** (S * K)
    n = N * (N - 1) / 2
    assert abs(c.sum() - q * n) < 5 * math.sqrt(n * q * (1 - q))
    # uniform over key positions: early and late halves of the causal range are hit alike
    m = oracle.mask_dense(spec)
    low = np.tril(np.ones((N, N), bool), -1)
    half = np.arange(N)[None, :] < (np.arange(N)[:, None] // 2)
    a, b = m[low & half].mean(), m[low & ~half].mean()
    assert abs(a - b) < 5 * math.sqrt(2 * q * (1 - q) / (low.sum() / 2))


def test_draw_sampler_union_and_edges(oracle):
    """Union over seeds is the OR of the per-seed draw masks; K = 0 leaves the forced set only;
    density 1 is dense causal whatever the sampler."""
    N, seeds = 300, [10, 20, 30]
    for mode in (oracle.MODE_STOCHASTIC, oracle.MODE_STRUCTURAL):
        u = oracle.mask_dense(oracle.MaskSpec(N=N, mode=mode, density=0.04, seeds=seeds, sampler=1))
        per = [oracle.mask_dense(oracle.MaskSpec(N=N, mode=mode, density=0.04, seeds=seeds, seed_index=s,
                                                 sampler=1)) for s in range(3)]
        np.testing.assert_array_equal(u, per[0] | per[1] | per[2])
        assert not (per[0] == per[1]).all()
    m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=0, density=0.001, seeds=[1], local_window=4, sampler=1))
    i, j = np.indices((N, N))
    np.testing.assert_array_equal(m, (j <= i) & (j > i - 4))
    m = oracle.mask_dense(oracle.MaskSpec(N=N, mode=0, density=1.0, seeds=[1], sampler=1))
    np.testing.assert_array_equal(m, np.tril(np.ones((N, N), bool)))
    a = oracle.mask_dense(oracle.MaskSpec(N=N, mode=0, density=0.05, seeds=[1], sampler=1))
    b = oracle.mask_dense(oracle.MaskSpec(N=N, mode=0, density=0.05, seeds=[1], sampler=0))
    assert (a != b).any()


# ----------------------------------------------------------------------------- Hybrid Anchor decode
def test_decode_anchor_matches_triton_bernoulli(oracle, tmp_path):
    """The Stochastic Anchor is row t0 = N of the prefill's RIS mask without its window: each
    j < t0 is kept iff some seed's Philox word (Triton's independent implementation, counter
    (j/4, t0, stream, layer_key), key (seed, head_key)) is below thr, plus the anchor tokens
    and, for Structural, the clique of t0's block."""
    pytest.importorskip("triton")
    N, seeds, A = 300, [4, 8], 3
    cases = [(oracle.MODE_STOCHASTIC, 0.05, 0, 0), (oracle.MODE_STRUCTURAL, 0.08, 1, 2)]
    for mode, d, hk, lk in cases:
        g = oracle.structural(N, d)
        p, stream = (g["d_global"], 1) if mode == oracle.MODE_STRUCTURAL else (d, 0)
        js = np.arange(N)
        ctr = np.array([(j // 4, N, stream, lk) for s in seeds for j in js], dtype=np.uint32)
        key = np.array([(s, hk) for s in seeds for j in js], dtype=np.uint32)
        words = _triton_philox(tmp_path, ctr, key).reshape(len(seeds), N, 4)
        u = words[:, js, js % 4]
        want = set(js[(u < oracle.threshold(p)).any(0)].tolist()) | set(range(A))
        if mode == oracle.MODE_STRUCTURAL:
            want |= set(range((N // g["B"]) * g["B"], N))
        spec = oracle.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, n_anchor=A, head_key=hk, layer_key=lk,
                               local_window=7)
        got = oracle.decode_anchor(spec)
        assert set(got.tolist()) == want and (np.diff(got) > 0).all() and got.max() < N


def test_decode_full_window_equals_dense_causal_row(oracle):
    """A window that reaches position 0 covers every earlier key: the decode output is the last
    row of dense causal attention (torch fp64 SDPA) over the rotated sequence."""
    N, t, Hq, Hkv, D = 64, 70, 4, 2, 32
    q, k, v = _rand((t + 1, Hq, D), 21), _rand((t + 1, Hkv, D), 22), _rand((t + 1, Hkv, D), 23)
    cfg = oracle.RopeCfg(kind=3, theta=1e4, native_len=32)
    anchor = oracle.decode_anchor(oracle.MaskSpec(N=N, mode=0, density=0.1, seeds=[1]))
    out, lse, keys = oracle.decode_step(q[t], k, v, t, anchor, window=t + 1, rope_cfg=cfg, n_ctx=N)
    np.testing.assert_array_equal(keys, np.arange(t + 1))
    pos = np.arange(t + 1, dtype=np.float64)
    qr, kr = oracle.rope(q, pos, cfg, N), oracle.rope(k, pos, cfg, N)
    ref, ref_lse = _sdpa(qr, kr, v, np.tril(np.ones((t + 1, t + 1), bool)), Hq // Hkv)
    np.testing.assert_allclose(out, ref[t], rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse[t], rtol=1e-12, atol=1e-12)


def test_decode_merge_is_set_union_with_one_softmax(oracle):
    """Window and anchor overlap: the key set is their set union (each key once), and the output
    is one softmax over it (brute force in torch fp64 on the explicit key rows)."""
    N, Hq, Hkv, D = 125, 6, 2, 16
    anchor = oracle.decode_anchor(oracle.MaskSpec(N=N, mode=1, density=0.1, seeds=[3, 5]))
    assert set(range(120, 125)) <= set(anchor.tolist())  # B = 12: t0 = 125 shares block [120, 132)
    for t, W in ((125, 16), (128, 1), (130, 30), (200, 5)):
        q, k, v = _rand((Hq, D), t), _rand((t + 1, Hkv, D), t + 1), _rand((t + 1, Hkv, D), t + 2)
        out, lse, keys = oracle.decode_step(q, k, v, t, anchor, W, None, N)
        want = sorted(set(anchor.tolist()) | set(range(max(0, t - W + 1), t + 1)))
        np.testing.assert_array_equal(keys, want)
        G = Hq // Hkv
        for h in range(Hq):
            kt = torch.from_numpy(k[keys, h // G])
            s = kt @ torch.from_numpy(q[h]) / math.sqrt(D)
            p = torch.softmax(s, 0)
            np.testing.assert_allclose(out[h], (p[:, None] * torch.from_numpy(v[keys, h // G])).sum(0).numpy(),
                                       rtol=1e-10, atol=1e-12)
            np.testing.assert_allclose(lse[h], torch.logsumexp(s, 0).item(), rtol=1e-12)
    out, _, _ = oracle.decode_step(q, k, np.ones_like(v), 200, anchor, 5, None, N)
    np.testing.assert_allclose(out, 1.0, atol=1e-13)
