"""Seeded random cases through the C ABI, as a net under the targeted tests.

Per-tensor calls: random shapes (ragged rows, all block sizes), methods
(ScaleSweep, AbsMax, 4/6), objectives, window modes (default, tight, custom),
input types, global scales and value distributions (including very small and
very large magnitudes and exact zeros) against the oracle with the near-tie rule.
Grouped calls: random groups of 1 to 16 tensors, static or dynamic scales,
against the per-tensor calls bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize

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


def draw(rng, rows, cols):
    kind = rng.integers(0, 5)
    if kind == 0:
        x = rng.standard_normal((rows, cols)) * 10.0 ** rng.uniform(-6, 3)
    elif kind == 1:
        x = rng.standard_t(2.5, (rows, cols))
    elif kind == 2:
        x = rng.laplace(0.0, 1.0, (rows, cols)) * np.exp(rng.standard_normal(cols))[None, :]
    elif kind == 3:                                   # sparse: many exact zeros, some zero blocks
        x = rng.standard_normal((rows, cols)) * (rng.random((rows, cols)) < 0.2)
    else:                                             # a few huge outlier channels
        x = rng.standard_normal((rows, cols)) * 0.01
        x[:, rng.integers(0, cols, 3)] *= 1e4
    return x.astype(np.float32)


@pytest.mark.parametrize("seed", range(64))
def test_random_per_tensor(B, seed):
    rng = np.random.default_rng(1000 + seed)
    block = int(rng.choice([16, 32, 64]))
    rows = int(rng.integers(1, 300))
    cols = block * int(rng.integers(1, 24))
    method = int(rng.choice([0, 0, 0, 1, 2]))
    obj = int(rng.integers(0, 2)) if method != 1 else 0
    dtype = torch.bfloat16 if rng.random() < 0.6 else torch.float32
    x = torch.from_numpy(draw(rng, rows, cols)).to(dtype)
    xs = x.float().numpy()
    D = float(rng.choice([256.0, 448.0, 6.0, 1e4]))
    S, _ = oracle.global_scale(xs, D)
    if rng.random() < 0.1:
        S = 0.0                                       # unusable scale: signs only
    w = torch.exp(torch.from_numpy(rng.standard_normal(cols).astype(np.float32))) if obj else None
    mode = int(rng.integers(0, 3)) if method == 0 else 0
    if mode == 0:
        win, owin = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT), None
    elif mode == 1:
        win, owin = (B.NVFP4_WINDOW_TIGHT, B.NVFP4_WINDOW_TIGHT), None     # same result as the default
    else:
        lo = int(rng.integers(-12, 1))
        hi = int(rng.integers(0, 12))
        win = owin = (lo, hi)
    xd = x.to(DEV)
    Sd = torch.tensor([S], dtype=torch.float32, device=DEV)
    swz = block == 16
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=swz, loss=True)
    wd = w.to(DEV) if w is not None else None
    if method == 0:
        B.scalesweep_quantize(xd, block, Sd, obj, wd, 0, *win, o["codes"], o["sf_linear"], o["sf_swizzled"],
                              o["block_loss"])
        ref = oracle.quantize(0, xs, block, S, obj, w=None if w is None else w.numpy(), window=owin)
    elif method == 1:
        B.absmax_quantize(xd, block, Sd, o["codes"], o["sf_linear"], o["sf_swizzled"], o["block_loss"])
        ref = oracle.quantize(1, xs, block, S, 0)
    else:
        B.four_over_six_quantize(xd, block, Sd, obj, wd, 0, o["codes"], o["sf_linear"], o["sf_swizzled"],
                                 o["block_loss"])
        ref = oracle.quantize(2, xs, block, S, obj, w=None if w is None else w.numpy())
    torch.cuda.synchronize()
    if method != 0:
        o["block_loss"] = None                        # baselines report their own losses; codes are the check
    compare_quantize(xs, S, block, obj, w, 0, o, ref)


@pytest.mark.parametrize("seed", range(24))
def test_random_groups(B, seed):
    rng = np.random.default_rng(2000 + seed)
    count = int(rng.integers(1, 17))
    obj = int(rng.integers(0, 2))
    dyn = rng.random() < 0.6
    dtype = torch.bfloat16 if rng.random() < 0.7 else torch.float32
    xs, ws, strides = [], [], []
    for _ in range(count):
        r = int(rng.integers(0, 200))
        c = 16 * int(rng.integers(1, 40))
        xs.append(torch.from_numpy(draw(rng, r, c)).to(dtype).to(DEV))
        if obj:
            if rng.random() < 0.3 and r > 0:
                stride = c + 4 * int(rng.integers(0, 3))
                ws.append(torch.exp(torch.from_numpy(rng.standard_normal((r, stride)).astype(np.float32))).to(DEV))
                strides.append(stride)
            else:
                ws.append(torch.exp(torch.from_numpy(rng.standard_normal(c).astype(np.float32))).to(DEV))
                strides.append(0)
        else:
            ws.append(None)
            strides.append(0)
    outs = [B.empty_outputs(x.shape[0], x.shape[1], 16, device=DEV, linear=True, swizzled=True) for x in xs]
    desc = B.group_descriptors(xs, ws, strides, [o["codes"] for o in outs], [o["sf_linear"] for o in outs],
                               [o["sf_swizzled"] for o in outs])
    dt = B.NVFP4_IN_BF16 if dtype == torch.bfloat16 else B.NVFP4_IN_F32
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    if dyn:
        S = torch.full((count,), -1.0, device=DEV)
        wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
        B.scalesweep_quantize_group(desc, dt, obj, 256.0, S, st, wsb)
    else:
        S = torch.tensor([float(rng.uniform(1e-4, 1.0)) for _ in range(count)], dtype=torch.float32, device=DEV)
        B.scalesweep_quantize_group(desc, dt, obj, 0.0, S, st, None)
    torch.cuda.synchronize()
    assert st.item() == 0
    for i, x in enumerate(xs):
        Si = torch.empty(1, device=DEV)
        if dyn:
            g = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
            B.nvfp4_global_scale(x, 256.0, Si, None, g)
            torch.cuda.synchronize()
            assert Si.item() == S[i].item()
        else:
            Si.copy_(S[i:i + 1])
        if x.numel() == 0:
            continue
        o = B.empty_outputs(x.shape[0], x.shape[1], 16, device=DEV, linear=True, swizzled=True)
        B.scalesweep_quantize(x, 16, Si, obj, ws[i], strides[i], *win, o["codes"], o["sf_linear"], o["sf_swizzled"])
        torch.cuda.synchronize()
        for k in ("codes", "sf_linear", "sf_swizzled"):
            assert torch.equal(o[k], outs[i][k]), (i, k)
