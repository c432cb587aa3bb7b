"""The default-window sweep skips low window offsets that a warp rules out with
a lower bound on their loss (the block's largest element's own error term).
That must not change anything: codes, both scale layouts and per-block losses
are compared bit for bit against the same window given explicitly, a call
that evaluates every candidate of the window with no skipping, on inputs that
stress the bound: heavy-tailed blocks (where the bound skips), blocks whose
largest value repeats, all-zero and NaN/inf blocks in the same warp, negative
and NaN weights (for which skipping must switch itself off), per-row weights,
global scales near the ends of the E4M3 range, and blocks of 16, 32 and 64 in
both input types.  The per-tensor sweep skips for MSE; the grouped launch,
which must give the same bytes, skips for MSE and for WMSE with blocks of 16.
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


def inputs(kind, rows, cols, seed):
    if kind == "laplace":                      # heavy-tailed, outlier channels: most low offsets are skipped
        x = W.small_tensor(rows, cols, seed, dist="laplace", std=0.015, outliers=max(1, cols // 200), mult=30.0)
    elif kind == "student_t":
        x = W.small_tensor(rows, cols, seed, dist="student_t", std=1.0, outliers=2, mult=50.0)
    elif kind == "repeated_max":               # every block's largest magnitude appears twice, with both signs
        x = W.small_tensor(rows, cols, seed, dist="normal", std=0.02).float()
        xb = x.view(rows, -1, 16)
        i = xb.abs().argmax(-1, keepdim=True)
        m = xb.abs().gather(-1, i)
        xb[..., 15:16] = -m
        xb.scatter_(-1, i, m)
        x = x.to(torch.bfloat16)
    else:                                      # mixed: zero, NaN and inf blocks among normal ones
        x = W.small_tensor(rows, cols, seed, dist="normal", std=0.02).float()
        x[0, :16] = 0.0
        x[1, 16:32] = float("nan")
        x[2, 32] = float("inf")
        x[3, 64:80] = 1e-30
        x = x.to(torch.bfloat16)
    return x


def weights(kind, rows, cols, seed):
    g = torch.Generator().manual_seed(seed)
    if kind == "per_row":
        return torch.exp(torch.randn(rows, cols + 4, generator=g)), cols + 4
    w = torch.exp(torch.randn(cols, generator=g))
    if kind == "negative":
        w[::7] *= -1.0                         # negative weights: the bound does not hold, no skipping
    elif kind == "nan":
        w[5] = float("nan")
    return w, 0


def run(B, x, block, S, obj, w, stride, window):
    rows, cols = x.shape
    out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16, loss=True)
    B.scalesweep_quantize(x, block, S, obj, w, stride, window[0], window[1], out["codes"], out["sf_linear"],
                          out["sf_swizzled"], out["block_loss"])
    torch.cuda.synchronize()
    return out


def run_group(B, x, block, S, obj, w, stride):
    rows, cols = x.shape
    out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16)
    desc = B.group_descriptors([x], [w], [stride], [out["codes"]], [out["sf_linear"]], [out["sf_swizzled"]])
    dt = B.NVFP4_IN_BF16 if x.dtype == torch.bfloat16 else B.NVFP4_IN_F32
    B.scalesweep_quantize_group(desc, dt, obj, 0.0, S, None, None, block=block)
    torch.cuda.synchronize()
    return out


def same(a, b):
    for k in ("codes", "sf_linear", "sf_swizzled", "block_loss"):
        if a[k] is None:
            continue
        if k == "block_loss":
            assert torch.equal(a[k].view(torch.int32), b[k].view(torch.int32)), k
        else:
            assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("obj,wkind", [(0, None), (1, "channel"), (1, "per_row"), (1, "negative"), (1, "nan")])
@pytest.mark.parametrize("xkind", ["laplace", "student_t", "repeated_max", "mixed"])
def test_skipping_sweep_equals_full_window(B, dtype, block, obj, wkind, xkind):
    rows, cols = 130, 1024
    x = inputs(xkind, rows, cols, 11 + block).to(dtype)
    xd = x.to(DEV)
    w, stride = weights(wkind, rows, cols, 5) if obj else (None, 0)
    wd = w.to(DEV) if w is not None else None
    lo = -3 if (obj == 0 and block == 16) else -8
    finite = x.float()[torch.isfinite(x.float())]
    for S_val in (float(oracle.global_scale(finite.numpy(), 256.0)[0]), 2.0 ** -100, 3.0e4):
        S = torch.tensor([S_val], dtype=torch.float32, device=DEV)
        fast = run(B, xd, block, S, obj, wd, stride, (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT))
        full = run(B, xd, block, S, obj, wd, stride, (lo, 7))
        same(fast, full)
        grouped = run_group(B, xd, block, S, obj, wd, stride)      # the grouped sweep skips for WMSE too
        for k in ("codes", "sf_linear", "sf_swizzled"):
            if grouped[k] is not None:
                assert torch.equal(grouped[k], full[k]), k


@pytest.mark.parametrize("obj", [0, 1])
@pytest.mark.parametrize("block", [16, 32, 64])
def test_skipping_sweep_matches_oracle_and_grouped_launch(B, obj, block):
    """Heavy-tailed weights (the Qwen2.5-72B recipe on 256 rows): the oracle's
    codes and scales (near-tie rule), and the grouped launch's bytes."""
    wl = W.workload("qwen72b-b16-wmse")
    t = wl.tensors[1]
    x = W.draw(t, rows=slice(0, 256))
    w = W.draw_weights(t) if obj else None
    xs = x.float().numpy()
    So, _ = oracle.global_scale(xs, 256.0)
    S = torch.tensor([So], dtype=torch.float32, device=DEV)
    xd = x.to(DEV)
    wd = w.to(DEV) if w is not None else None
    out = run(B, xd, block, S, obj, wd, 0, (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT))
    ref = oracle.quantize(0, xs, block, So, obj, w=None if w is None else w.numpy())
    compare_quantize(xs, So, block, obj, w, 0, out, ref)
    go = B.empty_outputs(x.shape[0], x.shape[1], block, device=DEV, linear=True, swizzled=block == 16)
    desc = B.group_descriptors([xd], [wd], [0], [go["codes"]], [go["sf_linear"]], [go["sf_swizzled"]])
    B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, obj, 0.0, S, None, None, block=block)
    torch.cuda.synchronize()
    for k in ("codes", "sf_linear", "sf_swizzled"):
        if go[k] is not None:
            assert torch.equal(go[k], out[k]), k
