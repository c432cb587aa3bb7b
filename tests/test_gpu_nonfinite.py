"""Blocks holding NaN or inf, and blocks whose normalised magnitude reaches
2^48, on the GPU: every entry point gives them the zero rule (scale code 0,
nibbles carrying only the sign of y) exactly as the oracle does, and every
other block of the tensor is unaffected.

The scale is static here (taken from the clean tensor) so that the planted
values reach the sweep; with a dynamic scale a NaN is skipped by the amax
(and flagged), while an inf makes S infinite and every block zero-ruled.
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


def planted(dtype, block, seed=11):
    """A clean tensor, its global scale, and a copy with one planted value in
    several small-magnitude blocks: NaN, +inf, -inf, a magnitude that puts
    y = fl(x E) at or above 2^48, and one near 2^47 (swept normally)."""
    rows, cols = 96, 4 * block * 3
    x = W.small_tensor(rows, cols, seed, dist="normal", std=0.02, outliers=2, mult=20.0).to(dtype)
    xf = x.float().numpy()
    S, _ = oracle.global_scale(xf, 256.0)
    E = np.float32(1) / np.float32(S)
    xp = x.clone()
    xp[3, block + 1] = float("nan")
    xp[10, 2 * block + 5] = float("inf")
    xp[17, 7] = float("-inf")
    xp[17, 8] = -0.0
    # smallest positive value of the input type with fl(x E) >= 2^48: step the
    # bit pattern upwards from just below 2^48 / E
    big = torch.tensor([2.0 ** 48 / float(E) * (1 - 2 ** -6)], dtype=torch.float32).to(dtype)
    ibits = torch.int16 if dtype == torch.bfloat16 else torch.int32
    while float(np.float32(big.float().item()) * E) < 2.0 ** 48:
        big = (big.view(ibits) + 1).view(dtype)
    xp[40, 3 * block + 2] = big[0]
    xp[41, block + 3] = torch.tensor(2.0 ** 47 / float(E), dtype=torch.float32).to(dtype)
    return xp, S


def run(B, method, x, block, S, obj, w):
    rows, cols = x.shape
    out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16)
    Sd = torch.tensor([S], dtype=torch.float32, device=DEV)
    xd = x.to(DEV)
    wd = None if w is None else w.to(DEV)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    if method == 0:
        B.scalesweep_quantize(xd, block, Sd, obj, wd, 0, *win, out["codes"], out["sf_linear"], out["sf_swizzled"],
                              None)
    elif method == 1:
        B.absmax_quantize(xd, block, Sd, out["codes"], out["sf_linear"], out["sf_swizzled"], None)
    else:
        B.four_over_six_quantize(xd, block, Sd, obj, wd, 0, out["codes"], out["sf_linear"], out["sf_swizzled"],
                                 None)
    torch.cuda.synchronize()
    return out


def zero_ruled(x, S, block):
    """Blocks the rule covers, from the inputs: max |fl(x E)| NaN, inf or >= 2^48."""
    y = (x.float().numpy() * (np.float32(1) / np.float32(S))).astype(np.float32)
    yb = np.abs(y.reshape(x.shape[0], -1, block))
    return np.isnan(yb).any(axis=2) | ~(np.nanmax(yb, axis=2) < 2.0 ** 48)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("method,obj", [(0, 0), (0, 1), (1, 0), (2, 0), (2, 1)])
def test_nonfinite_blocks_per_tensor(B, dtype, block, method, obj):
    xp, S = planted(dtype, block)
    cols = xp.shape[1]
    w = torch.exp(torch.randn(cols, generator=torch.Generator().manual_seed(2))) if obj == 1 else None
    out = run(B, method, xp, block, S, obj, w)
    xs = xp.float().numpy()
    wn = None if w is None else w.numpy()
    ref = oracle.quantize(method, xs, block, S, obj, w=wn, w_row_stride=0)
    compare_quantize(xs, S, block, obj, w, 0, out, ref, method=method)
    zr = zero_ruled(xp, S, block)
    assert zr.sum() == 4
    assert torch.all(out["sf_linear"].cpu()[torch.from_numpy(zr)] == 0)


@pytest.mark.parametrize("dyn", [False, True])
@pytest.mark.parametrize("obj", [0, 1])
def test_nonfinite_blocks_grouped(B, dyn, obj):
    """Grouped launch with two planted tensors and a clean one.  Static: the
    clean tensors' scales.  Dynamic: only NaN is planted (an inf would make S
    infinite), the scale skips it and bit 0 of the status word is set."""
    x0, S0 = planted(torch.bfloat16, 16, seed=21)
    x1, S1 = planted(torch.bfloat16, 16, seed=22)
    x2 = W.small_tensor(70, 128, 23).to(torch.bfloat16)
    S2, _ = oracle.global_scale(x2.float().numpy(), 256.0)
    if dyn:
        for x in (x0, x1):
            fin = ~torch.isfinite(x.float()) | (x.float().abs() > 1e3)
            x[fin] = 0.01
        x0[5, 20] = float("nan")
        x1[60, 40] = float("nan")
        x1[61, 41] = float("nan")
    xs = [x0, x1, x2]
    ws = [torch.exp(torch.randn(x.shape[1], generator=torch.Generator().manual_seed(7 + i))) if obj else None
          for i, x in enumerate(xs)]
    dx = [x.to(DEV) for x in xs]
    dw = [w.to(DEV) if w is not None else None for w in ws]
    outs = [B.empty_outputs(x.shape[0], x.shape[1], 16, device=DEV, linear=True, swizzled=True) for x in xs]
    desc = B.group_descriptors(dx, dw, [0, 0, 0], [o["codes"] for o in outs], [o["sf_linear"] for o in outs],
                               [o["sf_swizzled"] for o in outs])
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    if dyn:
        S = torch.full((3,), -1.0, device=DEV)
        gws = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
        B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, obj, 256.0, S, st, gws)
    else:
        S = torch.tensor([S0, S1, S2], dtype=torch.float32, device=DEV)
        B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, obj, 0.0, S, st, None)
    torch.cuda.synchronize()
    if dyn:
        assert st.item() & 1
    for i, x in enumerate(xs):
        xf = x.float().numpy()
        Si = float(S[i].item())
        if dyn:
            So, bad = oracle.global_scale(xf, 256.0)
            assert Si == np.float32(So) and bad == (i < 2)
        ref = oracle.quantize(0, xf, 16, Si, obj, w=None if ws[i] is None else ws[i].numpy())
        compare_quantize(xf, Si, 16, obj, ws[i], 0, outs[i], ref)
        if i < 2:
            zr = zero_ruled(x, Si, 16)
            assert zr.any() and torch.all(outs[i]["sf_linear"].cpu()[torch.from_numpy(zr)] == 0)


def test_nonfinite_blocks_fused_dynamic(B):
    """The fused dynamic-scale sweep: a NaN inside a small-magnitude block is
    skipped by the in-launch amax, flagged, and its block zero-ruled."""
    x = W.small_tensor(256, 512, 31).to(torch.bfloat16)
    x[9, 33] = float("nan")
    x[200, 500] = float("nan")
    xd = x.to(DEV)
    out = B.empty_outputs(256, 512, 16, device=DEV, linear=True, swizzled=True)
    S = torch.full((1,), -1.0, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=DEV)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    B.scalesweep_quantize_dynamic(xd, 16, 256.0, B.NVFP4_OBJ_MSE, None, 0, *win, S, st, ws, out["codes"],
                                  out["sf_linear"], out["sf_swizzled"], None)
    torch.cuda.synchronize()
    assert st.item() & 1
    xf = x.float().numpy()
    So, bad = oracle.global_scale(xf, 256.0)
    assert S.item() == np.float32(So) and bad
    ref = oracle.quantize(0, xf, 16, So, oracle.MSE)
    compare_quantize(xf, So, 16, 0, None, 0, out, ref)
    assert out["sf_linear"][9, 2].item() == 0 and out["sf_linear"][200, 31].item() == 0
