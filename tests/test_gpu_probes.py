"""Measurement-support calls on the GPU: ceiling probes and the library's memory-pool counters."""
import pytest
import torch

from paper_2607_21927_gb300 import ris

pytestmark = pytest.mark.gpu


def test_probes_are_plausible():
    l2 = ris.ris_probe_l2_bytes()
    assert 16 << 20 <= l2 <= 1 << 30
    stream_l2 = ris.ris_probe_l2_read(32 << 20, 0)
    rows_l2 = ris.ris_probe_l2_read(32 << 20, 1)
    hbm = ris.ris_probe_l2_read(4 * l2, 0)
    # an L2-resident working set streams faster than one four times the L2 size
    assert stream_l2 > hbm > 100.0
    assert rows_l2 > 100.0
    assert ris.ris_probe_ffma() > 1.0


def test_probe_rejects_bad_arguments():
    with pytest.raises(ris.RisError):
        ris.ris_probe_l2_read(1000, 0)
    with pytest.raises(ris.RisError):
        ris.ris_probe_l2_read(1 << 24, 7)


def test_memory_stats_track_mask():
    torch.cuda.synchronize()
    cur0, _ = ris.ris_memory_stats(reset_high_water=True)
    m = ris.ris_mask_generate(4096, 2, 0, 0.05, [0, 1, 2])
    torch.cuda.synchronize()
    cur1, high1 = ris.ris_memory_stats()
    d = m.info()
    held = d.n_pairs * d.col_bytes + (4096 + 1) * 8
    assert cur1 - cur0 >= held
    assert high1 >= cur1
    m.free()
    torch.cuda.synchronize()
    cur2, _ = ris.ris_memory_stats()
    assert cur2 <= cur1 - held
