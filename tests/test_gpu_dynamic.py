"""Fused dynamic-scale path (global scale computed inside the sweep launch).

It must reproduce the two-launch path (nvfp4_global_scale, then the sweep)
bit for bit -- S, codes, both scale layouts, per-block losses -- and so the
oracle; it must flag non-finite input and survive back-to-back calls on one
workspace (the grid-barrier counter is reset by the launch itself).
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


def two_launch(B, method, x, block, D, obj, w, win):
    rows, cols = x.shape
    S = torch.empty(1, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, D, S, st, ws)
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16, loss=True)
    if method == 0:
        B.scalesweep_quantize(x, block, S, obj, w, 0, *win, o["codes"], o["sf_linear"], o["sf_swizzled"],
                              o["block_loss"])
    else:
        B.absmax_quantize(x, block, S, o["codes"], o["sf_linear"], o["sf_swizzled"], o["block_loss"])
    return S, st, o


def fused(B, method, x, block, D, obj, w, win, ws=None):
    rows, cols = x.shape
    S = torch.full((1,), -1.0, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    if ws is None:
        ws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=DEV)
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16, loss=True)
    if method == 0:
        B.scalesweep_quantize_dynamic(x, block, D, obj, w, 0, *win, S, st, ws, o["codes"], o["sf_linear"],
                                      o["sf_swizzled"], o["block_loss"])
    else:
        B.absmax_quantize_dynamic(x, block, D, S, st, ws, o["codes"], o["sf_linear"], o["sf_swizzled"],
                                  o["block_loss"])
    return S, st, o


def same(a, b):
    for k in ("codes", "sf_linear", "sf_swizzled", "block_loss"):
        if a[k] is None:
            continue
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("rows,cols", [(1, 64), (130, 192), (2048, 1024), (8192, 4096)])
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("obj", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_fused_equals_two_launch(B, rows, cols, block, obj, dtype):
    x = W.small_tensor(rows, cols, rows + cols + block, dist="student_t", std=1.0, outliers=2, mult=50.0)
    xd = x.to(dtype).to(DEV)
    w = torch.exp(torch.randn(cols, generator=torch.Generator().manual_seed(rows))).to(DEV) if obj else None
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    for method in (0, 1):
        if method == 1 and obj == 1:
            continue
        S0, st0, o0 = two_launch(B, method, xd, block, 256.0, obj, w, win)
        S1, st1, o1 = fused(B, method, xd, block, 256.0, obj, w, win)
        torch.cuda.synchronize()
        assert S1.item() == S0.item() and st1.item() == st0.item() == 0
        same(o0, o1)


def test_fused_custom_window_and_oracle(B):
    x = W.small_tensor(300, 512, 5, dist="laplace", std=0.015, outliers=3, mult=30.0)
    xd = x.to(DEV)
    for win in ((-126, 126), (-1, 2)):
        S, st, o = fused(B, 0, xd, 16, 256.0, 0, None, win)
        torch.cuda.synchronize()
        xs = x.float().numpy()
        So, _ = oracle.global_scale(xs, 256.0)
        assert S.item() == np.float32(So)
        compare_quantize(xs, So, 16, 0, None, 0, o, oracle.quantize(0, xs, 16, So, 0, window=win))


def test_fused_activation_workload_full_size(B):
    """The per-call activation workload (8192 x 4096 Student-t, 16 outlier
    channels x50, MSE) through the fused path, sampled rows vs the oracle."""
    wl = W.workload("act-8192")
    t = wl.tensors[0]
    x = W.draw(t)
    S, st, o = fused(B, 0, x.to(DEV), 16, wl.fp8_div, 0, None, (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT))
    torch.cuda.synchronize()
    xs = x.float().numpy()
    So, _ = oracle.global_scale(xs, wl.fp8_div)
    assert S.item() == np.float32(So) and st.item() == 0
    idx = np.unique(np.linspace(0, t.rows - 1, 64).astype(np.int64))
    sub = {"codes": o["codes"][idx], "sf_linear": o["sf_linear"][idx],
           "block_loss": o["block_loss"].view(t.rows, -1)[idx].reshape(-1)}
    compare_quantize(xs[idx], So, 16, 0, None, 0, sub, oracle.quantize(0, xs[idx], 16, So, 0))


def test_fused_nonfinite_flag_and_reuse(B):
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    ws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=DEV)
    x = W.small_tensor(512, 1024, 3).to(DEV)
    ref = None
    for k in range(3):                               # the same workspace back to back
        S, st, o = fused(B, 0, x, 16, 256.0, 0, None, win, ws=ws)
        torch.cuda.synchronize()
        assert st.item() == 0
        if ref is None:
            ref = (S.item(), o)
        else:
            assert S.item() == ref[0]
            same(ref[1], o)
    bad = x.clone()
    bad[7, 9] = float("nan")
    S, st, o = fused(B, 0, bad, 16, 256.0, 0, None, win, ws=ws)
    torch.cuda.synchronize()
    assert st.item() & 1
    empty = torch.empty(0, 64, dtype=torch.bfloat16, device=DEV)
    S, st, o = fused(B, 0, empty, 16, 256.0, 0, None, win, ws=ws)
    torch.cuda.synchronize()
    assert S.item() == -1.0 and st.item() == 0         # nothing launched for an empty input
