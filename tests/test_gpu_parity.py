"""GPU parity: the CUDA library, called through its C ABI, against the CPU oracle.

Codes and scales must be bit-exact except on oracle near-ties (see
tests/parity.py); global scales and dequantised tensors are bit-exact; per-block
and summed losses agree to fp32 accumulation accuracy (1e-5 relative summed).
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize, to_np, x_to_f32
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


def gscale(B, x, D):
    S = torch.empty(1, dtype=torch.float32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, D, S, st, ws)
    return S, st


def quant(B, method, x, block, S, obj=0, w=None, stride=0, window=None, swz=None, loss=True):
    rows, cols = x.shape
    if swz is None:
        swz = block == 16
    out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=swz, loss=loss)
    if method == 0:
        lo, hi = window if window is not None else (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
        B.scalesweep_quantize(x, block, S, obj, w, stride, lo, hi, out["codes"], out["sf_linear"],
                              out["sf_swizzled"], out["block_loss"])
    elif method == 1:
        B.absmax_quantize(x, block, S, out["codes"], out["sf_linear"], out["sf_swizzled"], out["block_loss"])
    else:
        B.four_over_six_quantize(x, block, S, obj, w, stride, out["codes"], out["sf_linear"], out["sf_swizzled"],
                                 out["block_loss"])
    torch.cuda.synchronize()
    return out


def oracle_quant(method, xs, block, S, obj, w, stride, window=None):
    wn = None if w is None else to_np(w)
    if method == 0:
        return oracle.quantize(0, xs, block, S, obj, w=wn, w_row_stride=stride, window=window)
    return oracle.quantize(method, xs, block, S, obj if method == 2 else 0, w=wn if method == 2 else None,
                           w_row_stride=stride)


# --------------------------------------------------------------------------- global scale
@pytest.mark.parametrize("n", [1, 7, 8, 9, 1000, 4 * 1024 * 1024 + 3])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_global_scale_bit_exact(B, n, dtype):
    g = torch.Generator().manual_seed(n)
    x = (torch.randn(n, generator=g) * 3).to(dtype)
    xd = x.to(DEV)
    for D in (448.0, 256.0):
        S, st = gscale(B, xd, D)
        So, bad = oracle.global_scale(x.float().numpy(), D)
        assert S.item() == np.float32(So) and st.item() == 0 and not bad


def test_global_scale_nonfinite_flag(B):
    x = torch.randn(100003, dtype=torch.float32)
    x[5] = float("nan")
    S, st = gscale(B, x.to(DEV), 256.0)
    assert st.item() == 1 and S.item() == np.float32(oracle.global_scale(x.numpy(), 256.0)[0])
    x[7] = float("-inf")
    S, st = gscale(B, x.to(DEV), 256.0)
    assert st.item() == 1 and np.isinf(S.item())
    z = torch.zeros(64, dtype=torch.bfloat16, device=DEV)
    S, st = gscale(B, z, 256.0)
    assert S.item() == 0.0 and st.item() == 0


# --------------------------------------------------------------------------- small shapes
SHAPES = [(1, 64), (3, 128), (33, 256), (130, 192), (257, 64)]


@pytest.mark.parametrize("rows,cols", SHAPES)
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("method", [0, 1, 2])
@pytest.mark.parametrize("obj", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_quantize_small_shapes(B, rows, cols, block, method, obj, dtype):
    if method == 1 and obj == 1:
        pytest.skip("AbsMax has no objective")
    seed = rows * 1000 + cols + block + 7 * method + 3 * obj
    dist = ["normal", "student_t", "laplace"][seed % 3]
    x = W.small_tensor(rows, cols, seed, dist=dist, std=0.02, outliers=2, mult=25.0).to(dtype)
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 256.0)
    w, stride = None, 0
    if obj == 1:
        g = torch.Generator().manual_seed(seed + 1)
        if seed % 2:
            w = torch.exp(torch.randn(cols, generator=g)).to(DEV)
        else:
            w, stride = torch.exp(torch.randn(rows, cols, generator=g)).to(DEV), cols
    gpu = quant(B, method, xd, block, S, obj, w, stride)
    ref = oracle_quant(method, x.float().numpy(), block, S.item(), obj, w, stride)
    compare_quantize(x.float().numpy(), S.item(), block, obj if method != 1 else 0, w, stride, gpu, ref, method)


# --------------------------------------------------------------------------- edge cases
def test_zero_blocks_signed_zero_and_zero_tensor(B):
    x = W.small_tensor(8, 64, 5).float()
    x[2, 16:32] = 0.0
    x[2, 20] = -0.0
    x[5, :] = -0.0
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 256.0)
    gpu = quant(B, 0, xd, 16, S)
    compare_quantize(x.numpy(), S.item(), 16, 0, None, 0, gpu, oracle.quantize(0, x.numpy(), 16, S.item()))
    z = torch.zeros(4, 32, device=DEV)
    z[1, 3] = -0.0
    Sz, _ = gscale(B, z, 256.0)
    gpu = quant(B, 0, z, 16, Sz)
    compare_quantize(z.cpu().numpy(), 0.0, 16, 0, None, 0, gpu, oracle.quantize(0, z.cpu().numpy(), 16, 0.0))


@pytest.mark.parametrize("Sval", [0.0, -1.0, float("inf"), float("nan"), 1e-40])
def test_unusable_global_scale(B, Sval):
    x = W.small_tensor(4, 64, 9).float()
    S = torch.tensor([Sval], dtype=torch.float32, device=DEV)
    for method in (0, 1, 2):
        gpu = quant(B, method, x.to(DEV), 16, S)
        ref = oracle.quantize(method, x.numpy(), 16, Sval)
        assert np.array_equal(to_np(gpu["sf_linear"]), ref["sf"])
        assert np.array_equal(to_np(gpu["codes"]), ref["codes"])


def test_tiny_and_saturating_blocks(B):
    g = torch.Generator().manual_seed(3)
    x = torch.randn(16, 128, generator=g)
    x[0] *= 1e-6          # block maxima far below 2^-9 * 6 S: I0 = 0 region
    x[1] *= 1e-4
    x[2, :16] = torch.linspace(-1e-7, 1e-7, 16)
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 256.0)
    for method in (0, 1, 2):
        gpu = quant(B, method, xd, 16, S)
        compare_quantize(x.numpy(), S.item(), 16, 0, None, 0, gpu, oracle.quantize(method, x.numpy(), 16, S.item()))
    # a static global scale far below amax/(6*448): every block saturates at 448
    Ssat = torch.tensor([float(x.abs().max()) / 6 / 448 / 50], device=DEV)
    for method in (0, 1, 2):
        gpu = quant(B, method, xd, 16, Ssat)
        compare_quantize(x.numpy(), Ssat.item(), 16, 0, None, 0, gpu,
                         oracle.quantize(method, x.numpy(), 16, Ssat.item()))


def test_window_edge_blocks_and_custom_windows(B):
    from test_oracle_sweep import EDGE_BLOCKS
    one = torch.ones(1, device=DEV)
    for obj, _, yv, wv in EDGE_BLOCKS:
        y = torch.tensor([yv], dtype=torch.float32)
        w = None if wv is None else torch.tensor(wv, dtype=torch.float32, device=DEV)
        gpu = quant(B, 0, y.to(DEV), 16, one, obj, w, 0)
        ref = oracle.quantize(0, y.numpy(), 16, 1.0, obj, w=None if wv is None else np.array(wv, np.float32))
        compare_quantize(y.numpy(), 1.0, 16, obj, w, 0, gpu, ref)
    x = W.small_tensor(64, 256, 77, dist="laplace", std=0.015, outliers=3, mult=30.0)
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 256.0)
    for win in ((-126, 126), (0, 0), (-1, 1), (-8, 7), (2, 30), (-126, -100)):
        gpu = quant(B, 0, xd, 16, S, window=win)
        ref = oracle.quantize(0, x.float().numpy(), 16, S.item(), 0, window=win)
        compare_quantize(x.float().numpy(), S.item(), 16, 0, None, 0, gpu, ref)


def test_exhaustive_equals_bounded_on_gpu(B):
    """Bounded = exhaustive (Sec. 4.2.2) on the 2048x2048 N(0, 0.02^2) matrix,
    D = 448, both computed by the GPU and both checked against the oracle."""
    x = W.draw(W.workload("weight-2048").tensors[0])
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 448.0)
    a = quant(B, 0, xd, 16, S)
    e = quant(B, 0, xd, 16, S, window=(-126, 126))
    assert torch.equal(a["sf_linear"], e["sf_linear"]) and torch.equal(a["codes"], e["codes"])
    xs = x.float().numpy()
    compare_quantize(xs, S.item(), 16, 0, None, 0, a, oracle.quantize(0, xs, 16, S.item()))


def test_output_guard_bytes_untouched(B):
    rows, cols, block = 130, 192, 16
    x = W.small_tensor(rows, cols, 12).to(DEV)
    S, _ = gscale(B, x, 256.0)
    G = 4096
    codes = torch.full((2 * G + rows * cols // 2,), 0xAB, dtype=torch.uint8, device=DEV)
    sfl = torch.full((2 * G + rows * cols // block,), 0xAB, dtype=torch.uint8, device=DEV)
    nsw = B.swizzled_bytes(rows, cols)
    sfs = torch.full((2 * G + nsw,), 0xAB, dtype=torch.uint8, device=DEV)
    loss = torch.full((2 * G + rows * cols // block,), 1.5, dtype=torch.float32, device=DEV)
    cv = codes[G:G + rows * cols // 2].view(rows, cols // 2)
    B.scalesweep_quantize(x, block, S, 0, None, 0, B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT, cv,
                          sfl[G:G + rows * cols // block], sfs[G:G + nsw], loss[G:G + rows * cols // block])
    torch.cuda.synchronize()
    for buf, n in ((codes, rows * cols // 2), (sfl, rows * cols // block), (sfs, nsw)):
        assert torch.all(buf[:G] == 0xAB) and torch.all(buf[G + n:] == 0xAB)
    n = rows * cols // block
    assert torch.all(loss[:G] == 1.5) and torch.all(loss[G + n:] == 1.5)


def test_bad_inputs_rejected_before_launch(B):
    x = W.small_tensor(8, 64, 1).to(DEV)
    S, _ = gscale(B, x, 256.0)
    out = B.empty_outputs(8, 64, 16, device=DEV, swizzled=True)
    args = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    xv = x.view(-1)[1:1 + 8 * 48].view(8, 48)          # 2-byte offset: misaligned
    with pytest.raises(B.Nvfp4Error) as ei:
        B.scalesweep_quantize(xv, 16, S, 0, None, 0, *args, out["codes"][:, :24], out["sf_linear"][:, :3])
    assert ei.value.code == 3
    with pytest.raises(B.Nvfp4Error) as ei:
        B.scalesweep_quantize(x.cpu(), 16, S, 0, None, 0, *args, out["codes"], out["sf_linear"])
    assert ei.value.code == 1                           # pageable host memory is not accepted
    with pytest.raises(B.Nvfp4Error) as ei:
        B.scalesweep_quantize(x, 32, S, 0, None, 0, *args, out["codes"], None, out["sf_swizzled"])
    assert ei.value.code == 2
    with pytest.raises(B.Nvfp4Error) as ei:
        B.scalesweep_quantize(x, 16, S, 0, None, 0, *args, out["codes"], out["codes"].view(-1)[:32])
    assert ei.value.code == 1
    torch.cuda.synchronize()


def test_dynamic_scale_on_side_stream_and_determinism(B):
    x = W.small_tensor(512, 512, 21, dist="student_t", std=1.0, outliers=4, mult=50.0).to(DEV)
    s = torch.cuda.Stream()
    outs = []
    for _ in range(2):
        with torch.cuda.stream(s):
            S = torch.empty(1, device=DEV)
            ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
            B.nvfp4_global_scale(x, 256.0, S, None, ws, stream=s)
            o = B.empty_outputs(512, 512, 16, device=DEV, swizzled=True, loss=True)
            B.scalesweep_quantize(x, 16, S, 0, None, 0, B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT, o["codes"],
                                  o["sf_linear"], o["sf_swizzled"], o["block_loss"], stream=s)
        s.synchronize()
        outs.append((S.clone(), o))
    assert torch.equal(outs[0][1]["codes"], outs[1][1]["codes"])
    assert torch.equal(outs[0][1]["block_loss"], outs[1][1]["block_loss"])
    xs = x_to_f32(x)
    compare_quantize(xs, outs[0][0].item(), 16, 0, None, 0, outs[0][1], oracle.quantize(0, xs, 16, outs[0][0].item()))


# --------------------------------------------------------------------------- dequantisation
@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("S_val", [0.0371, 1e-39, 3e36])     # ordinary; subnormal S; products past fp32/bf16 max
def test_dequantize_bit_exact(B, block, out_dtype, S_val):
    rows, cols = 131, 256
    g = np.random.default_rng(block)
    codes = g.integers(0, 256, (rows, cols // 2), dtype=np.uint8)
    sf = g.integers(0, 127, (rows, cols // block), dtype=np.uint8)
    S = np.float32(S_val)
    Sd = torch.tensor([S], device=DEV)
    layouts = [(1, sf)] + ([(2, oracle.swizzle_scales(sf))] if block == 16 else [])
    for layout, sfl in layouts:
        out = torch.empty(rows, cols, dtype=out_dtype, device=DEV)
        B.nvfp4_dequantize(torch.from_numpy(codes).to(DEV), torch.from_numpy(sfl).to(DEV), layout, Sd, rows, cols,
                           block, out)
        torch.cuda.synchronize()
        want = oracle.dequantize(codes, sfl, layout, float(S), rows, cols, block, out_bf16=out_dtype == torch.bfloat16)
        got = out.cpu().view(torch.int16).numpy().view(np.uint16) if out_dtype == torch.bfloat16 else \
            out.cpu().numpy().view(np.uint32)
        assert np.array_equal(got, want.view(got.dtype))


def test_quantize_dequantize_roundtrip_tensor_mse(B):
    """Summed tensor MSE from the GPU's dequantised output agrees with the
    oracle's float64 objective (x domain) to 1e-5 relative."""
    x = W.small_tensor(256, 1024, 31, dist="laplace", std=0.015, outliers=4, mult=30.0)
    xd = x.to(DEV)
    S, _ = gscale(B, xd, 256.0)
    gpu = quant(B, 0, xd, 16, S)
    out = torch.empty(256, 1024, device=DEV)
    B.nvfp4_dequantize(gpu["codes"], gpu["sf_swizzled"], 2, S, 256, 1024, 16, out)
    torch.cuda.synchronize()
    ref = oracle.quantize(0, x.float().numpy(), 16, S.item())
    xh = oracle.dequantize(ref["codes"], ref["sf"], 1, S.item(), 256, 1024, 16)
    assert np.array_equal(out.cpu().numpy().view(np.uint32), xh.view(np.uint32))
    mse_gpu = float(((out.double().cpu() - x.double()) ** 2).sum())
    mse_ref = float(ref["best"].sum()) * float(S.item()) ** 2
    assert abs(mse_gpu - mse_ref) <= 1e-5 * mse_ref
