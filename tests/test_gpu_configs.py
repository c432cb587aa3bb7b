"""Full-size parity on every synthetic workload, in the launch configuration
bench.py times (whole tensors, default windows, both scale layouts).

The GPU quantises each whole tensor; the oracle recomputes a sample of rows
(first, last and evenly spread ones) with the same S; every other block is
checked through properties that hold at any size (scale codes in the window
range, swizzled = permuted linear, dequantised values bounded by the block's
own scale).  The global scale is compared bit-exactly on the whole tensor.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize, to_np
from paper_2606_07618_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"
SAMPLE_ROWS = 48


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_07618_gb300 import binding
    binding.lib()
    oracle.build()
    return binding


_cache = {}


def tensors_of(name):
    wl = W.workload(name)
    key = tuple((t.seed, t.rows, t.cols) for t in wl.tensors)
    if key not in _cache:
        _cache.clear()
        _cache[key] = [(t, W.draw(t), W.draw_weights(t)) for t in wl.tensors]
    return wl, _cache[key]


def sample_rows(rows):
    idx = np.unique(np.concatenate([[0, rows - 1], np.linspace(0, rows - 1, SAMPLE_ROWS).astype(np.int64)]))
    return idx


@pytest.mark.parametrize("name", W.ALL_CONFIGS)
def test_workload_parity_full_size(B, name):
    wl, ts = tensors_of(name)
    obj = B.NVFP4_OBJ_WMSE if wl.objective == "wmse" else B.NVFP4_OBJ_MSE
    block = wl.block
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    for t, x, w in ts:
        xd = x.to(DEV)
        S = torch.empty(1, device=DEV)
        st = torch.zeros(1, dtype=torch.int32, device=DEV)
        ws = torch.empty(B.nvfp4_global_scale_workspace(xd.numel()), dtype=torch.uint8, device=DEV)
        B.nvfp4_global_scale(xd, wl.fp8_div, S, st, ws)
        xs = x.float().numpy()
        So, bad = oracle.global_scale(xs, wl.fp8_div)
        assert S.item() == np.float32(So) and st.item() == 0 and not bad

        rows, cols = x.shape
        out = B.empty_outputs(rows, cols, block, device=DEV, linear=True, swizzled=block == 16, loss=True)
        wd = w.to(DEV) if obj == B.NVFP4_OBJ_WMSE else None
        B.scalesweep_quantize(xd, block, S, obj, wd, 0, *win, out["codes"], out["sf_linear"], out["sf_swizzled"],
                              out["block_loss"])
        torch.cuda.synchronize()

        # sampled rows against the oracle (same S, same weights)
        idx = sample_rows(rows)
        sub = {"codes": out["codes"][idx], "sf_linear": out["sf_linear"][idx],
               "block_loss": out["block_loss"].view(rows, -1)[idx].reshape(-1)}
        wn = w.numpy() if obj == B.NVFP4_OBJ_WMSE else None
        ref = oracle.quantize(0, xs[idx], block, So, obj, w=wn, w_row_stride=0)
        compare_quantize(xs[idx], So, block, obj, wd, 0, sub, ref)

        # properties of every block
        sf = out["sf_linear"]
        assert int(sf.max()) <= 126
        if out["sf_swizzled"] is not None:
            kb = cols // 16
            r = torch.arange(rows, device=DEV).view(-1, 1)
            k = torch.arange(kb, device=DEV).view(1, -1)
            kpad4 = (kb + 3) // 4
            off = ((r // 128) * kpad4 + k // 4) * 512 + (r % 32) * 16 + ((r // 32) % 4) * 4 + (k % 4)
            assert torch.equal(out["sf_swizzled"][off.view(-1)].view(rows, kb), sf)
        # reconstruction stays within half a grid step of the clipped value: |x_hat| <= 6 s S and finite
        deq = torch.empty(rows, cols, device=DEV)
        B.nvfp4_dequantize(out["codes"], sf, B.NVFP4_SF_LINEAR, S, rows, cols, block, deq)
        vals = torch.from_numpy(np.array([oracle.e4m3_value(c) for c in range(127)] + [0.0] * 129,
                                         dtype=np.float32)).to(DEV)
        smax = (vals[sf.long()] * 6.0 * S).repeat_interleave(block, dim=1)
        assert torch.isfinite(deq).all()
        assert torch.all(deq.abs() <= smax * (1 + 1e-6))
        # total loss of the tensor equals the sum of the per-block losses (x domain)
        tot = float(((deq.double() - xd.double()) ** 2 * (wd.double() if wd is not None else 1.0)).sum())
        est = float(out["block_loss"].double().sum()) * float(S.item()) ** 2
        assert abs(tot - est) <= 1e-4 * est
        del xd, out, deq, smax
        torch.cuda.empty_cache()
