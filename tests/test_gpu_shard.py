"""The row partition on one GPU: N shards quantised one after another, with
the max-allreduce emulated by the maximum of the shards' [S bits, status]
pairs (the reduction the collective performs), write exactly the bytes of the
single whole-tensor call -- S, status, codes, linear and swizzled scales --
and match the oracle.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize
from paper_2606_07618_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_07618_gb300 import binding
    binding.lib()
    oracle.build()
    return binding


def whole_call(B, x, block, obj, w, D):
    rows, cols = x.shape
    S = torch.empty(1, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, D, S, st, ws)
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    B.scalesweep_quantize(x, block, S, obj, w, 0, *win, o["codes"], o["sf_linear"], o["sf_swizzled"], None)
    return S, st, o


def sharded_calls(B, x, block, obj, w, D, world):
    from paper_2606_07618_gb300 import shard
    rows, cols = x.shape
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16)
    for v in o.values():                        # poison: every byte must be written by some shard
        if v is not None:
            v.fill_(0xEE)
    lays = [shard.layout(rows, cols, block, world, r) for r in range(world)]
    bufs = [shard.scale(x[l.row_begin:l.row_end], D) for l in lays]
    red = torch.stack(bufs).max(dim=0).values.contiguous()          # what the MAX-allreduce yields
    for l in lays:
        shard.sweep(x[l.row_begin:l.row_end], red, block, obj, w, 0, shard.output_views(o, l))
    return shard.global_scale_of(red), red[1:2], o


@pytest.mark.parametrize("world", [2, 3, 8])
@pytest.mark.parametrize("shape,block,obj", [((4096, 4096), 16, 1), ((1000, 512), 16, 0), ((777, 320), 64, 1),
                                             ((300, 256), 32, 0), ((129, 64), 16, 1)])
def test_shards_equal_the_single_call(B, world, shape, block, obj):
    rows, cols = shape
    x = W.small_tensor(rows, cols, rows + cols, dist="laplace", std=0.015, outliers=2, mult=30.0).to(DEV)
    w = torch.exp(torch.randn(cols, generator=torch.Generator().manual_seed(cols))).to(DEV) if obj else None
    S1, st1, o1 = whole_call(B, x, block, obj, w, 256.0)
    S2, st2, o2 = sharded_calls(B, x, block, obj, w, 256.0, world)
    torch.cuda.synchronize()
    assert S1.item() == S2.item() and st1.item() == st2.item() == 0
    for k in ("codes", "sf_linear", "sf_swizzled"):
        if o1[k] is not None:
            assert torch.equal(o1[k], o2[k]), k
    xs = x.float().cpu().numpy()
    So, _ = oracle.global_scale(xs, 256.0)
    assert S2.item() == np.float32(So)
    ref = oracle.quantize(0, xs, block, So, obj, w=None if w is None else w.cpu().numpy())
    compare_quantize(xs, So, block, obj, w, 0, {k: v.cpu() if v is not None else None for k, v in o2.items()}, ref)


def test_shard_flags_and_empty_shards(B):
    """A NaN in one shard reaches every shard's status through the reduction;
    with more shards than 128-row blocks some shards are empty."""
    x = W.small_tensor(300, 128, 9).to(DEV)
    x[250, 3] = float("nan")
    S1, st1, o1 = whole_call(B, x, 16, 0, None, 256.0)
    S2, st2, o2 = sharded_calls(B, x, 16, 0, None, 256.0, 5)     # 3 row blocks over 5 shards
    torch.cuda.synchronize()
    assert st1.item() == 1 and st2.item() == 1 and S1.item() == S2.item()
    for k in ("codes", "sf_linear", "sf_swizzled"):
        assert torch.equal(o1[k], o2[k]), k
