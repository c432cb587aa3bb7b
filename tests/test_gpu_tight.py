"""The per-block tight window (NVFP4_WINDOW_TIGHT) on the GPU.

It must give the oracle's default-window result (the tight window only drops
candidates the paper proves cannot win; near-tie rule of parity.py) and the
GPU's own default-window result bit for bit outside near-ties, for both
objectives, blocks 16/32/64, bf16 and fp32, global scales that put I0 in the
normal range, at the top (448) and in the subnormal codes; through the
dynamic-scale entry point as well; and on the full 8192 x 4096 activation
workload (sampled rows against the oracle).
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize
from paper_2606_07618_gb300 import workloads as W
from test_gpu_parity import gscale, quant

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


def tight(B):
    return (B.NVFP4_WINDOW_TIGHT, B.NVFP4_WINDOW_TIGHT)


@pytest.mark.parametrize("obj,block", [(0, 16), (1, 16), (0, 32), (1, 64)])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("D", [256.0, 448.0, 0.05])
def test_tight_equals_default_and_oracle(B, obj, block, dtype, D):
    x = W.small_tensor(130, 512, 40 + block + obj, dist="student_t", std=1.0, outliers=3, mult=30.0).to(dtype)
    xd = x.to(DEV)
    w = torch.exp(torch.randn(512, generator=torch.Generator().manual_seed(block))).to(DEV) if obj else None
    S, _ = gscale(B, xd, D)
    t = quant(B, 0, xd, block, S, obj, w, 0, window=tight(B))
    d = quant(B, 0, xd, block, S, obj, w, 0)
    xs = x.float().numpy()
    ref = oracle.quantize(0, xs, block, S.item(), obj, w=None if w is None else w.cpu().numpy())
    compare_quantize(xs, S.item(), block, obj, w, 0, t, ref)
    diff = (t["sf_linear"] != d["sf_linear"]).sum().item()
    best, second = ref["best"], ref["second"]
    near = int(np.sum((second - best) <= 1e-6 * np.abs(best)))
    assert diff <= near


def test_tight_dynamic_entry_point(B):
    x = W.small_tensor(256, 1024, 9, dist="laplace", std=0.015, outliers=4, mult=30.0).to(DEV)
    S, _ = gscale(B, x, 256.0)
    a = quant(B, 0, x, 16, S, 0, None, 0, window=tight(B))
    o = B.empty_outputs(256, 1024, 16, device=DEV, linear=True, swizzled=True, loss=True)
    S2 = torch.empty(1, device=DEV)
    ws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=DEV)
    B.scalesweep_quantize_dynamic(x, 16, 256.0, 0, None, 0, *tight(B), S2, None, ws, o["codes"], o["sf_linear"],
                                  o["sf_swizzled"], o["block_loss"])
    torch.cuda.synchronize()
    assert S2.item() == S.item()
    for k in ("codes", "sf_linear", "sf_swizzled", "block_loss"):
        assert torch.equal(a[k], o[k]), k


def test_tight_full_size_activation(B):
    wl = W.workload("act-8192")
    t = wl.tensors[0]
    x = W.draw(t)
    xd = x.to(DEV)
    S, _ = gscale(B, xd, wl.fp8_div)
    a = quant(B, 0, xd, 16, S, 0, None, 0, window=tight(B), loss=False)
    d = quant(B, 0, xd, 16, S, 0, None, 0, loss=False)
    differ = (a["sf_linear"] != d["sf_linear"]).sum().item()
    assert differ <= a["sf_linear"].numel() // 100000
    idx = np.unique(np.linspace(0, t.rows - 1, 48).astype(np.int64))
    xs = x.float().numpy()[idx]
    sub = {"codes": a["codes"][idx], "sf_linear": a["sf_linear"][idx]}
    compare_quantize(xs, S.item(), 16, 0, None, 0, sub, oracle.quantize(0, xs, 16, S.item(), 0))
