"""GPU optimal FP32 block scale and FP8-quantised optimum (Appendix C) against
the oracle's sorted-breakpoint enumeration in float64.

The optimum is a continuous minimum, so losses are compared (fp32 result to
1e-5 relative); the GPU's s_opt must attain its reported loss when the loss is
re-evaluated exactly at that s; the FP8-quantised code must equal the oracle's
except where s_opt sits at an E4M3 value or the two rounded candidates tie.
Invariants: optimum <= ScaleSweep's loss per block; for MSE with 16-element
blocks ScaleSweep <= the FP8-quantised optimum (the window holds the optimum).
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
    from paper_2606_07618_gb300 import binding
    binding.lib()
    oracle.build()
    return binding


def exact_loss(a, w, s):
    a = np.abs(a.astype(np.float64))
    g = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6])
    q = g[np.argmin(np.abs(a[:, None] / s - g[None, :]), axis=1)]
    return float(np.sum((1.0 if w is None else w.astype(np.float64)) * (a - s * q) ** 2))


@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("obj", [0, 1])
@pytest.mark.parametrize("dist", ["normal", "student_t", "laplace"])
def test_optimal_scale_matches_oracle(B, block, obj, dist):
    rows, cols = 24, 256
    x = W.small_tensor(rows, cols, block * 7 + obj, dist=dist, std=0.02 if dist == "normal" else 1.0, outliers=2,
                       mult=30.0)
    xd = x.to(DEV)
    S = torch.empty(1, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(xd.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(xd, 256.0, S, None, ws)
    w = torch.exp(torch.randn(cols, generator=torch.Generator().manual_seed(block))).to(DEV) if obj else None
    nb = rows * cols // block
    s_opt = torch.empty(nb, device=DEV)
    l_opt = torch.empty(nb, device=DEV)
    code = torch.empty(nb, dtype=torch.uint8, device=DEV)
    l_fp8 = torch.empty(nb, device=DEV)
    B.nvfp4_optimal_scale(xd, block, S, obj, w, 0, s_opt, l_opt, code, l_fp8)
    out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, loss=True)
    B.scalesweep_quantize(xd, block, S, obj, w, 0, B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT, out["codes"],
                          out["sf_linear"], None, out["block_loss"])
    torch.cuda.synchronize()
    Sv = S.item()
    E = np.float32(1) / np.float32(Sv)
    y = (x.float().numpy() * E).astype(np.float32).reshape(rows, -1, block)
    wn = None if w is None else w.cpu().numpy()
    so, lo, co, lf = (to.cpu().numpy() for to in (s_opt, l_opt, code, l_fp8))
    ss = out["block_loss"].cpu().numpy()
    for r in range(rows):
        for k in range(cols // block):
            b = r * (cols // block) + k
            wb = None if wn is None else wn[k * block:(k + 1) * block]
            s_ref, L_ref = oracle.opt_scale(y[r, k], wb)
            assert abs(lo[b] - L_ref) <= 1e-5 * L_ref + 1e-30, (b, lo[b], L_ref)
            if so[b] > 0:
                Lg = exact_loss(y[r, k], wb, float(so[b]))
                assert Lg <= lo[b] * (1 + 1e-5) + 1e-30 and Lg >= L_ref * (1 - 1e-9)
            s_use = s_ref
            if so[b] > 0 and abs(so[b] - s_ref) > 1e-5 * s_ref:
                # several scales attain the optimum; score the FP8 rounding of the GPU's one
                assert abs(exact_loss(y[r, k], wb, float(so[b])) - L_ref) <= 1e-6 * L_ref
                s_use = float(so[b])
            c_ref, Lf_ref = oracle.fp8_opt_code(y[r, k], wb, s_use)
            if co[b] != c_ref:
                # only where s_opt sits on an E4M3 value or floor/ceil tie
                v = [oracle.e4m3_value(c) for c in (co[b], c_ref)]
                near = min(abs(s_use - vv) for vv in v) <= 1e-5 * s_use
                assert near or abs(lf[b] - Lf_ref) <= 1e-5 * Lf_ref, (b, co[b], c_ref)
            assert abs(lf[b] - Lf_ref) <= 1e-5 * Lf_ref + 1e-30 or co[b] != c_ref
            assert lo[b] <= ss[b] * (1 + 1e-5) + 1e-30
            if obj == 0 and block == 16:
                assert ss[b] <= lf[b] * (1 + 1e-5) + 1e-30
