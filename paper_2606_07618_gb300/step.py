"""One pass of the hot path over a set of tensors, through the C ABI.

``QuantizeStep`` owns the output buffers for a list of tensors and
quantises all of them with ONE library call per step: the per-call global
scale of every tensor (S = amax / (6 D), Sec. 4.2.1) and the ScaleSweep of
every block (Sec. 4.2.2), writing packed E2M1 codes and E4M3 scales.

  * several tensors, or a single weight: ``scalesweep_quantize_group`` with
    in-launch scales (a layer's weights, the KV-cache/query tensors, ...);
  * a single activation tensor (``activation=True``): the fused
    ``scalesweep_quantize_dynamic`` (amax and sweep in one cooperative launch).

``absmax`` runs the AbsMax baseline (Sec. 3.2) over the same tensors in the
same launch shape, so the two can be compared call for call.  Every step runs
on the GPU in the library's kernels; this module only arranges buffers and
arguments.
"""
from __future__ import annotations

import torch

from . import binding as B


class QuantizeStep:
    def __init__(self, xs, ws=None, block: int = 16, objective: int = B.NVFP4_OBJ_MSE, fp8_div: float = 256.0,
                 activation: bool = False, swizzled: bool | None = None, w_row_strides=None, outs=None,
                 device=None):
        """xs: tensors the GPU can read (device memory, or pinned host memory
        the kernels then read over the host link); outs: optional output dicts
        as from binding.empty_outputs (e.g. pinned host memory), else device
        buffers are allocated; device: where S, the status word and the
        workspace live (default: the device of xs[0])."""
        if not xs:
            raise ValueError("QuantizeStep needs at least one tensor")
        self.xs = list(xs)
        self.ws = list(ws) if ws is not None else [None] * len(self.xs)
        self.block = int(block)
        self.objective = int(objective)
        self.fp8_div = float(fp8_div)
        self.fused = bool(activation) and len(self.xs) == 1
        dev = torch.device(device) if device is not None else self.xs[0].device
        if swizzled is None:
            swizzled = self.block == 16
        self.outs = list(outs) if outs is not None else [
            B.empty_outputs(x.shape[0], x.shape[1], self.block, device=dev, linear=True, swizzled=swizzled)
            for x in self.xs]
        self.S = torch.empty(len(self.xs), dtype=torch.float32, device=dev)
        self.status = torch.zeros(1, dtype=torch.int32, device=dev)
        self.dtype = B.NVFP4_IN_BF16 if self.xs[0].dtype == torch.bfloat16 else B.NVFP4_IN_F32
        strides = list(w_row_strides) if w_row_strides is not None else [0] * len(self.xs)
        self.strides = strides
        if self.fused:
            self.workspace = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=dev)
        else:
            self.workspace = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=dev)
            self.desc = B.group_descriptors(self.xs, self.ws, strides, [o["codes"] for o in self.outs],
                                            [o["sf_linear"] for o in self.outs],
                                            [o["sf_swizzled"] for o in self.outs])

    @property
    def numel(self) -> int:
        return sum(x.numel() for x in self.xs)

    @property
    def pipelined(self) -> bool:
        """Whether the grouped call takes the pipelined schedule (the library's
        choice: a ScaleSweep over at least two tensors and 2^25 elements)."""
        return not self.fused and len(self.xs) >= 2 and self.numel >= 1 << 25

    def __call__(self, stream=None):
        """ScaleSweep over every tensor (one library call: a workspace memset,
        then one cooperative launch or the pipelined schedule's four)."""
        if self.fused:
            o = self.outs[0]
            win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
            B.scalesweep_quantize_dynamic(self.xs[0], self.block, self.fp8_div, self.objective, self.ws[0],
                                          self.strides[0], *win, self.S, self.status, self.workspace, o["codes"],
                                          o["sf_linear"], o["sf_swizzled"], None, stream=stream)
        else:
            B.scalesweep_quantize_group(self.desc, self.dtype, self.objective, self.fp8_div, self.S, self.status,
                                        self.workspace, stream=stream, block=self.block)

    def absmax(self, stream=None):
        """The AbsMax baseline over the same tensors, same launch shape."""
        if self.fused:
            o = self.outs[0]
            B.absmax_quantize_dynamic(self.xs[0], self.block, self.fp8_div, self.S, self.status, self.workspace,
                                      o["codes"], o["sf_linear"], o["sf_swizzled"], None, stream=stream)
        else:
            B.absmax_quantize_group(self.desc, self.dtype, self.fp8_div, self.S, self.status, self.workspace,
                                    stream=stream, block=self.block)


def for_workload(wl, xs, ws=None) -> QuantizeStep:
    """The launch configuration of a synthetic workload (workloads.py)."""
    obj = B.NVFP4_OBJ_WMSE if wl.objective == "wmse" else B.NVFP4_OBJ_MSE
    return QuantizeStep(xs, ws if obj == B.NVFP4_OBJ_WMSE else None, block=wl.block, objective=obj,
                        fp8_div=wl.fp8_div, activation=wl.dynamic_scale)
