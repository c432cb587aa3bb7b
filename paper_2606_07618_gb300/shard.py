"""Row-sharded quantisation of one tensor over the ranks of a process group.

Given the global scale S, every block is independent (Sec. 4.2.1), so a
[rows, cols] tensor can be split by rows across GPUs.  The only exchange is
the per-call global scale: each rank reduces its own rows' amax into
S_k = fl32(amax_k / fl32(6 D)) with nvfp4_global_scale, and one
max-allreduce gives every rank S = max_k S_k, which is the whole tensor's S
bit for bit (fl32(a / c) is monotone in a).  The status words (bit 0: NaN or
inf seen) are reduced in the same collective: both values sit in one int32
pair, and for the non-negative S (finite or +inf, never NaN) the order of the
bit patterns is the order of the values, so one MAX reduces both.

nvfp4_row_shard_layout puts shard boundaries on multiples of 128 rows, so
every shard's codes, linear scales and 128x4 swizzled-scale atoms are
contiguous byte ranges of the whole tensor's outputs: a rank's outputs are
either its own buffers or views at those offsets into full-size buffers.

    lay = shard.layout(rows, cols, block, world, rank)
    buf = shard.scale(x_rows, fp8_div)              # this rank's S_k and status
    shard.allreduce_scale(buf, group)               # the one collective
    shard.sweep(x_rows, buf, block, objective, w, w_row_stride, outs)

Every compute step runs in the library's kernels; the collective is
torch.distributed (NCCL across GPUs, gloo on CPU in the tests).
"""
from __future__ import annotations

import torch

from . import binding as B


def layout(rows: int, cols: int, block: int, world: int, rank: int) -> B.RowShard:
    """Rows [row_begin, row_end) and output offsets of shard `rank`."""
    return B.nvfp4_row_shard_layout(rows, cols, block, world, rank)


def output_views(outs: dict, lay: B.RowShard) -> dict:
    """The shard's slices of full-size outputs from binding.empty_outputs
    (codes [rows, cols/2], sf_linear [rows, kb], sf_swizzled flat bytes)."""
    r0, r1 = lay.row_begin, lay.row_end
    v = {"codes": outs["codes"][r0:r1], "sf_linear": None, "sf_swizzled": None}
    if outs.get("sf_linear") is not None:
        v["sf_linear"] = outs["sf_linear"][r0:r1]
    if outs.get("sf_swizzled") is not None and lay.sf_swizzled_offset >= 0:
        v["sf_swizzled"] = outs["sf_swizzled"][lay.sf_swizzled_offset:lay.sf_swizzled_offset + lay.sf_swizzled_bytes]
    return v


def scale(x_rows: torch.Tensor, fp8_div: float, workspace: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """int32[2] on x's device: the bits of this shard's S_k and its status word
    (an empty shard contributes S_k = 0, status 0)."""
    buf = torch.zeros(2, dtype=torch.int32, device=x_rows.device)
    if x_rows.numel():
        if workspace is None:
            workspace = torch.empty(B.nvfp4_global_scale_workspace(x_rows.numel()), dtype=torch.uint8,
                                    device=x_rows.device)
        B.nvfp4_global_scale(x_rows, fp8_div, buf[0:1].view(torch.float32), buf[1:2], workspace, stream=stream)
    return buf


def allreduce_scale(buf: torch.Tensor, group=None) -> torch.Tensor:
    """The partition's one exchange: MAX-allreduce of [S bits, status] across
    the group (in place); a no-op without an initialised process group."""
    import torch.distributed as dist
    if dist.is_available() and dist.is_initialized() and dist.get_world_size(group) > 1:
        dist.all_reduce(buf, op=dist.ReduceOp.MAX, group=group)
    return buf


def global_scale_of(buf: torch.Tensor) -> torch.Tensor:
    """The reduced S as a one-element float32 view of buf."""
    return buf[0:1].view(torch.float32)


def sweep(x_rows: torch.Tensor, buf: torch.Tensor, block: int, objective: int, w, w_row_stride: int, outs: dict,
          stream=None):
    """ScaleSweep of this shard's rows with the reduced S (default window)."""
    if x_rows.numel() == 0:
        return
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    B.scalesweep_quantize(x_rows, block, global_scale_of(buf), objective, w, w_row_stride, *win, outs["codes"],
                          outs.get("sf_linear"), outs.get("sf_swizzled"), None, stream=stream)


def quantize_rows(x_rows: torch.Tensor, block: int, objective: int, w, w_row_stride: int, fp8_div: float, outs: dict,
                  group=None, stream=None) -> torch.Tensor:
    """scale -> allreduce_scale -> sweep for this rank's rows; returns buf."""
    buf = scale(x_rows, fp8_div, stream=stream)
    allreduce_scale(buf, group)
    sweep(x_rows, buf, block, objective, w, w_row_stride, outs, stream=stream)
    return buf
