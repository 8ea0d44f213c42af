"""Rank-split of one AF1 layer over G GPUs (one exchange step).

y = a * (U (s * (V^T (b * x)))) is a sum over the rank index k, so GPU g can
hold the columns k in [r0, r1) of U and V (and s[r0:r1]), with a and b
replicated, and compute the partial y_g = a * U_g (s_g * (V_g^T (b * x))).
The layer output is the sum of the G partials: one all-reduce (sum) of
tokens x m FP32 values per call. Every GPU streams about 1/G of the packed
signs. Slices start on 128-rank boundaries, so a slice of the canonical
packed words is a contiguous range of whole words (U, packed along r) or of
whole rows (V^T, one row per rank index).

Host-side bookkeeping only: each GPU runs the library's own forward on its
slice; torch.distributed provides the all-reduce.
"""
from __future__ import annotations

import torch


def words_per_row(cols: int) -> int:
    """32-bit words of one canonical packed row (16-byte padded)."""
    return 4 * ((cols + 127) // 128)


def rank_slices(r: int, world: int) -> list[tuple[int, int]]:
    """[r0, r1) per GPU: as equal as 128-rank granularity allows; a GPU may
    get an empty slice when r has fewer 128-blocks than GPUs."""
    if world < 1 or r < 1:
        raise ValueError("world and r must be >= 1")
    blocks = (r + 127) // 128
    out, b0 = [], 0
    for g in range(world):
        nb = blocks // world + (1 if g < blocks % world else 0)
        r0, r1 = min(128 * b0, r), min(128 * (b0 + nb), r)
        out.append((r0, r1))
        b0 += nb
    return out


def slice_packed(Uw: torch.Tensor, Vw: torch.Tensor, s: torch.Tensor, r0: int, r1: int):
    """Canonical packed words and rank scales of ranks [r0, r1).

    Uw: (m, W(r)) words of U (packed along r); Vw: (r, W(n)) words of V^T;
    s: (r,) rank scales. r0 must be a multiple of 128. The last slice keeps
    the zero padding bits of the original rows."""
    if r0 % 128 != 0 or not (0 <= r0 < r1):
        raise ValueError("slices start on a multiple of 128 and are non-empty")
    w0, wn = r0 // 32, words_per_row(r1 - r0)
    Uw_g = Uw[:, w0:w0 + wn]
    if Uw_g.shape[1] < wn:  # cannot happen for canonical rows; kept explicit
        pad = torch.zeros((Uw.shape[0], wn - Uw_g.shape[1]), dtype=Uw.dtype, device=Uw.device)
        Uw_g = torch.cat([Uw_g, pad], dim=1)
    return Uw_g.contiguous(), Vw[r0:r1].contiguous(), s[r0:r1].contiguous()


def forward_rank_split(layer_g, x: torch.Tensor, y32: torch.Tensor, workspace: torch.Tensor, group=None,
                       stream=None, host_reduce: bool = False) -> torch.Tensor:
    """This GPU's partial (FP32) followed by the all-reduce (sum) over the
    process group; y32 (tokens, m) float32 holds the layer output on return.
    host_reduce: all-reduce a host copy (for process groups whose backend
    reduces host tensors, e.g. gloo) and copy the sum back."""
    import torch.distributed as dist
    if layer_g is None:
        y32.zero_()  # a GPU without ranks contributes zeros
    else:
        layer_g.forward_into(x, y32, workspace, stream=stream)
    if host_reduce:
        if stream is not None:
            stream.synchronize()
        yh = y32.cpu()
        dist.all_reduce(yh, op=dist.ReduceOp.SUM, group=group)
        y32.copy_(yh)
    else:
        dist.all_reduce(y32, op=dist.ReduceOp.SUM, group=group)
    return y32
