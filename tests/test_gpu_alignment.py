"""Inputs that are 16-byte but not 32-byte aligned, and the global-scale
launches captured in a CUDA graph.

The C ABI asks for 16-byte aligned inputs only; an input that starts 16 bytes
past a 32-byte boundary must give the codes, scales and losses of the same
values at an aligned address bit for bit (and so the oracle's), for every
method, objective, block size and input type, through the per-tensor,
dynamic-scale and grouped entry points.  The global scale's second launch is a
programmatic dependent of the first; captured in a graph and replayed on new
data it must give the exact amax / (6 D) of that data.
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


def offset16(x):
    """A copy of x whose data starts 16 bytes past a 32-byte boundary."""
    k = 16 // x.element_size()
    buf = torch.empty(x.numel() + 2 * k, dtype=x.dtype, device=x.device)
    if buf.data_ptr() % 32 != 0:
        pytest.skip("allocator returned a base that is not 32-byte aligned")
    v = buf[k:k + x.numel()].view(x.shape)
    v.copy_(x)
    assert v.data_ptr() % 32 == 16
    return v


def gscale(B, x, D=256.0):
    S = torch.empty(1, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, D, S, None, ws)
    return S


def run(B, method, x, block, S, obj, w):
    rows, cols = x.shape
    o = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16, loss=True)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    if method == 0:
        B.scalesweep_quantize(x, block, S, obj, w, 0, *win, o["codes"], o["sf_linear"], o["sf_swizzled"],
                              o["block_loss"])
    elif method == 1:
        B.absmax_quantize(x, block, S, o["codes"], o["sf_linear"], o["sf_swizzled"], o["block_loss"])
    else:
        B.four_over_six_quantize(x, block, S, obj, w, 0, o["codes"], o["sf_linear"], o["sf_swizzled"],
                                 o["block_loss"])
    torch.cuda.synchronize()
    return o


@pytest.mark.parametrize("method,obj", [(0, 0), (0, 1), (1, 0), (2, 1)])
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_sixteen_byte_aligned_input_per_tensor(B, method, obj, block, dtype):
    x = W.small_tensor(67, 320, 5 + block, dist="student_t", std=1.0, outliers=3, mult=30.0).to(dtype).to(DEV)
    w = torch.exp(torch.randn(320, generator=torch.Generator().manual_seed(2))).to(DEV) if obj else None
    S = gscale(B, x)
    a = run(B, method, x, block, S, obj, w)
    xo = offset16(x)
    b = run(B, method, xo, block, S, obj, w)
    for k in ("codes", "sf_linear", "sf_swizzled", "block_loss"):
        if a[k] is not None:
            assert torch.equal(a[k], b[k]), k
    if method == 0:
        xs = x.float().cpu().numpy()
        ref = oracle.quantize(0, xs, block, S.item(), obj, w=None if w is None else w.cpu().numpy())
        compare_quantize(xs, S.item(), block, obj, w, 0, b, ref)


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_sixteen_byte_aligned_input_dynamic(B, dtype):
    x = W.small_tensor(300, 512, 17, dist="laplace", std=0.015, outliers=4, mult=30.0).to(dtype).to(DEV)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    outs, Ss = [], []
    for xx in (x, offset16(x)):
        o = B.empty_outputs(300, 512, 16, device=DEV, linear=True, swizzled=True, loss=True)
        S = torch.empty(1, device=DEV)
        ws = torch.empty(B.nvfp4_dynamic_workspace(), dtype=torch.uint8, device=DEV)
        B.scalesweep_quantize_dynamic(xx, 16, 256.0, 0, None, 0, *win, S, None, ws, o["codes"], o["sf_linear"],
                                      o["sf_swizzled"], o["block_loss"])
        torch.cuda.synchronize()
        outs.append(o)
        Ss.append(S.item())
    assert Ss[0] == Ss[1] == np.float32(oracle.global_scale(x.float().cpu().numpy(), 256.0)[0])
    for k in ("codes", "sf_linear", "sf_swizzled", "block_loss"):
        assert torch.equal(outs[0][k], outs[1][k]), k


@pytest.mark.parametrize("dyn", [False, True])
def test_sixteen_byte_aligned_input_group(B, dyn):
    shapes = [(200, 256), (33, 512), (128, 96)]
    xs = [W.small_tensor(r, c, 30 + i, dist="normal", std=0.02, outliers=2, mult=20.0).to(DEV)
          for i, (r, c) in enumerate(shapes)]
    ws = [torch.exp(torch.randn(c, generator=torch.Generator().manual_seed(i))).to(DEV)
          for i, (_, c) in enumerate(shapes)]
    res = []
    for inputs in (xs, [xs[0], offset16(xs[1]), offset16(xs[2])]):
        outs = [B.empty_outputs(r, c, 16, device=DEV, linear=True, swizzled=True) for r, c in shapes]
        desc = B.group_descriptors(inputs, ws, [0, 0, 0], [o["codes"] for o in outs],
                                   [o["sf_linear"] for o in outs], [o["sf_swizzled"] for o in outs])
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        if dyn:
            S = torch.empty(len(shapes), device=DEV)
            wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
            B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, 1, 256.0, S, st, wsb)
        else:
            S = torch.tensor([0.01, 0.002, 0.05], device=DEV)
            B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, 1, 0.0, S, st, None)
        torch.cuda.synchronize()
        assert st.item() == 0
        res.append((S.clone(), outs))
    assert torch.equal(res[0][0], res[1][0])
    for a, b in zip(res[0][1], res[1][1]):
        for k in ("codes", "sf_linear", "sf_swizzled"):
            assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_global_scale_and_sweep_in_cuda_graph(B, dtype):
    """Both global-scale launches (the fold a programmatic dependent of the
    partial maxima) and the sweep after them, captured once and replayed on
    new data in the captured input buffer."""
    rows, cols = 256, 1024
    x = torch.empty(rows, cols, dtype=dtype, device=DEV)
    S = torch.zeros(1, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    o = B.empty_outputs(rows, cols, 16, device=DEV, linear=True, swizzled=True)
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)

    def step(s):
        B.nvfp4_global_scale(x, 256.0, S, st, ws, stream=s)
        B.scalesweep_quantize(x, 16, S, 0, None, 0, *win, o["codes"], o["sf_linear"], o["sf_swizzled"], stream=s)

    x.copy_(W.small_tensor(rows, cols, 1).to(dtype))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        step(s)                                       # warm-up outside the capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        step(s)
    for seed, scale in ((11, 1.0), (12, 1e-3), (13, 40.0)):
        xc = (W.small_tensor(rows, cols, seed, dist="student_t", std=1.0, outliers=3, mult=30.0) * scale).to(dtype)
        x.copy_(xc.to(DEV))
        o["codes"].zero_()
        torch.cuda.synchronize()
        g.replay()
        torch.cuda.synchronize()
        xs = xc.float().numpy()
        So = oracle.global_scale(xs, 256.0)[0]
        assert S.item() == np.float32(So) and st.item() == 0
        ref = oracle.quantize(0, xs, 16, S.item(), 0)
        compare_quantize(xs, S.item(), 16, 0, None, 0, {"codes": o["codes"], "sf_linear": o["sf_linear"]}, ref)
