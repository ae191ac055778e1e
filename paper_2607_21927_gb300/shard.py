"""Query-row sharding of one prefill layer across ranks, each holding only its own rows.

Rows are independent given K, V and the counter-based mask (every rank builds the same mask
from the same seeds: the paper's master mask, Methods, "Memory-Bounded Geometry Generation"),
so one layer splits into contiguous row ranges of equal sampled-pair count
(ris_mask_row_split). A rank that holds only its own rows of q, k and v first all-gathers the
layer's K and V, its one exchange per layer, then attends its rows with
ris_attention_masked_local. The exchange goes through torch.distributed (NCCL between GPUs,
gloo on CPU); no kernel reads another device's memory.
"""
from __future__ import annotations

from typing import Optional, Sequence

import torch


def kv_allgather(k_rows: torch.Tensor, v_rows: torch.Tensor, bounds: Sequence[int], group=None):
    """Full K and V [N, Hkv, D] on this rank from every rank's rows bounds[r] .. bounds[r+1]-1.

    Parts may differ in length; each is padded to the longest for one all-gather of K and one
    of V, then the padding is dropped. Returns freshly allocated contiguous tensors.
    """
    import torch.distributed as dist

    world = dist.get_world_size(group)
    rank = dist.get_rank(group)
    assert len(bounds) == world + 1 and bounds[0] == 0
    n_mine = bounds[rank + 1] - bounds[rank]
    assert k_rows.shape[0] == n_mine and v_rows.shape == k_rows.shape
    longest = max(bounds[r + 1] - bounds[r] for r in range(world))
    full = []
    for x in (k_rows, v_rows):
        send = torch.zeros((longest,) + tuple(x.shape[1:]), dtype=x.dtype, device=x.device)
        send[:n_mine] = x
        parts = [torch.empty_like(send) for _ in range(world)]
        dist.all_gather(parts, send, group=group)
        full.append(torch.cat([parts[r][: bounds[r + 1] - bounds[r]] for r in range(world)], 0).contiguous())
    return full[0], full[1]


def attend_rows(mask, bounds: Sequence[int], rank: int, q_rows: torch.Tensor, k_full: torch.Tensor,
                v_full: torch.Tensor, rope=None, out_rows: Optional[torch.Tensor] = None, out_dtype=None):
    """This rank's rows of the layer output (ris_attention_masked_local)."""
    from . import ris

    return ris.ris_attention_masked_local(mask, bounds[rank], bounds[rank + 1], q_rows, k_full, v_full,
                                          out_rows=out_rows, rope=rope, out_dtype=out_dtype)
