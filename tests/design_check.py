"""Run a few attention cases through the C ABI under the kernel design named by
RIS_FORCE_DESIGN and compare them with the fp64 oracle; exit status 0 if all pass.
Invoked by tests/test_gpu_designs.py in a fresh process per design."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
sys.path.insert(0, os.path.dirname(os.path.abspath(__file__)))

import torch  # noqa: E402

import oracle  # noqa: E402
from helpers import check_bf16_path, make_inputs, to_np  # noqa: E402
from paper_2607_21927_gb300 import ris  # noqa: E402

CASES = [
    # N, Hq, Hkv, D, mode, density, seeds, rope (kind, theta, native) or None, per_seed
    (300, 6, 2, 128, 0, 0.05, [1, 2], (3, 1e6, 128), False),
    (700, 12, 2, 128, 0, 0.5, [1, 2], (1, 1e6, 32768), False),
    (257, 4, 1, 128, 2, 1.0, [0], None, False),
    (640, 8, 2, 64, 1, 0.1, [3], (2, 1e4, 128), False),
    (400, 6, 2, 128, 0, 0.3, [4, 5, 6], (3, 1e6, 256), True),
    (3, 6, 2, 128, 0, 0.5, [1], (3, 1e6, 64), False),
    (1, 2, 1, 64, 1, 0.5, [2], None, False),
    # Structural blocks of 300 and 260 tokens: the dense-suffix split (blocks on the tiles) where allowed
    (3000, 6, 2, 128, 1, 0.1, [1], (3, 1e6, 256), False),
    (2600, 4, 1, 128, 1, 0.12, [3], None, False),
]


def main():
    for N, Hq, Hkv, D, mode, d, seeds, rk, per_seed in CASES:
        (q, k, v), (qn, kn, vn) = make_inputs(N, Hq, Hkv, D, seed=N + len(seeds), outliers=True)
        rope = ris.rope_cfg(*rk) if rk else None
        fn = ris.ris_ensemble_batch if per_seed else ris.ris_sparse_attention_fwd
        out = fn(q, k, v, mode, d, seeds, rope=rope, out_dtype=torch.float32)
        ris.ris_device_status()
        cfg = oracle.RopeCfg(kind=rk[0], theta=rk[1], native_len=rk[2]) if rk else None
        for si in (range(len(seeds)) if per_seed else [-1]):
            spec = oracle.MaskSpec(N=N, mode=mode, density=d, seeds=seeds, seed_index=si)
            ref, _, _, _ = oracle.sparse_attention(qn, kn, vn, spec, cfg)
            got = to_np(out[si] if per_seed else out)
            err, rel = check_bf16_path(got, ref)
            print(f"{os.environ.get('RIS_FORCE_DESIGN')} N={N} H={Hq}/{Hkv} D={D} mode={mode} d={d} set={si}: "
                  f"max-abs {err:.2e} rel-L2 {rel:.2e}", flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
