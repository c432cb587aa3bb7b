"""Pin of the 128x4 swizzled scale layout (and of the packed E2M1 nibble order)
against NVIDIA's block-scaled GEMM: torch._scaled_mm with float4_e2m1fn_x2
operands and float8_e4m3fn block scales runs cuBLASLt's NVFP4 path, which reads
the scales in that layout.  The paper does not define the layout, so this
library routine is the independent reference for both the CUDA output and the
oracle's swizzle_scales.  A negative control (linear bytes passed as swizzled)
must fail, showing the check can tell layouts apart.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2606_07618_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if not hasattr(torch, "float4_e2m1fn_x2"):
        pytest.skip("torch without float4_e2m1fn_x2")
    from paper_2606_07618_gb300 import binding
    binding.lib()
    oracle.build()
    return binding


def quantize(B, x):
    S = torch.empty(1, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, 256.0, S, None, ws)
    o = B.empty_outputs(x.shape[0], x.shape[1], 16, device=DEV, linear=True, swizzled=True)
    B.scalesweep_quantize(x, 16, S, 0, None, 0, B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT, o["codes"],
                          o["sf_linear"], o["sf_swizzled"])
    d = torch.empty(x.shape[0], x.shape[1], device=DEV)
    B.nvfp4_dequantize(o["codes"], o["sf_linear"], B.NVFP4_SF_LINEAR, S, x.shape[0], x.shape[1], 16, d)
    torch.cuda.synchronize()
    return o, S, d


def nvfp4_gemm(codes_a, sf_a, codes_b, sf_b):
    return torch._scaled_mm(codes_a.view(torch.float4_e2m1fn_x2), codes_b.view(torch.float4_e2m1fn_x2).t(),
                            sf_a.view(torch.float8_e4m3fn), sf_b.view(torch.float8_e4m3fn),
                            out_dtype=torch.float32).double()


@pytest.mark.parametrize("M,N,K", [(256, 384, 512), (128, 128, 2048), (512, 256, 1024)])
def test_swizzled_scales_drive_cublaslt_nvfp4_gemm(B, M, N, K):
    a = W.small_tensor(M, K, M + K, dist="normal", std=1.0).to(DEV)
    b = W.small_tensor(N, K, N + K + 1, dist="laplace", std=0.5, outliers=2, mult=20.0).to(DEV)
    oa, Sa, da = quantize(B, a)
    ob, Sb, db = quantize(B, b)
    ref = (da.double() @ db.double().T) / (Sa.double() * Sb.double())   # q*s products, global scales removed
    scale = ref.abs().max().item()
    try:
        got = nvfp4_gemm(oa["codes"], oa["sf_swizzled"], ob["codes"], ob["sf_swizzled"])
    except (RuntimeError, NotImplementedError) as e:
        pytest.skip(f"NVFP4 _scaled_mm unavailable: {e}")
    assert (got - ref).abs().max().item() <= 1e-6 * scale
    # the oracle's layout function, applied to the GPU's linear scales, drives the same GEMM
    sfa_o = torch.from_numpy(oracle.swizzle_scales(oa["sf_linear"].cpu().numpy())).to(DEV)
    sfb_o = torch.from_numpy(oracle.swizzle_scales(ob["sf_linear"].cpu().numpy())).to(DEV)
    got_o = nvfp4_gemm(oa["codes"], sfa_o, ob["codes"], sfb_o)
    assert (got_o - ref).abs().max().item() <= 1e-6 * scale
    # negative control: linear bytes in place of the swizzled layout
    lin_a = torch.zeros_like(oa["sf_swizzled"])
    lin_a[:oa["sf_linear"].numel()] = oa["sf_linear"].view(-1)
    lin_b = torch.zeros_like(ob["sf_swizzled"])
    lin_b[:ob["sf_linear"].numel()] = ob["sf_linear"].view(-1)
    bad = nvfp4_gemm(oa["codes"], lin_a, ob["codes"], lin_b)
    assert (bad - ref).abs().max().item() > 1e-2 * scale
