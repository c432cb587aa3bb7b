"""Full-size parity on every synthetic workload, every block, in the launch
configuration bench.py times (paper_2606_07618_gb300.step: one grouped launch
with in-launch global scales, or the fused dynamic launch for the activation).

For every tensor of every workload -- the 2048x2048 weight, the Llama-3-8B
layer, the 8192x4096 activation, K/V/Q, and both Qwen2.5-72B-shaped matrices
at blocks 16/32/64 with MSE and WMSE:

  * S equals the oracle's bit for bit;
  * every block's scale and nibbles equal the oracle's, except on the
    oracle's near-ties (best and second-best within 1e-6 relative), where the
    GPU's pick must score within 1e-6 of the best and carry the oracle's
    nibbles for that scale (tests/parity.py);
  * the dequantised tensor equals the oracle's dequantisation of the same
    codes bit for bit (swizzled scales for block 16, linear otherwise);
  * the tensor's summed loss, measured on the GPU from its own output in the
    x domain, agrees with the oracle's summed block optimum times S^2 to 1e-5.

The per-workload counts (blocks checked, near-ties accepted) are printed.
"""
import os

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


_cache = {}


def tensors_of(name):
    wl = W.workload(name)
    key = tuple((t.seed, t.rows, t.cols) for t in wl.tensors)
    if key not in _cache:
        _cache.clear()
        _cache[key] = [(t, W.draw(t), W.draw_weights(t)) for t in wl.tensors]
    return wl, _cache[key]


def _threads():
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)


@pytest.mark.parametrize("name", W.ALL_CONFIGS)
def test_workload_parity_every_block(B, name, capsys):
    from paper_2606_07618_gb300 import step as ST
    wl, ts = tensors_of(name)
    wmse = wl.objective == "wmse"
    obj = B.NVFP4_OBJ_WMSE if wmse else B.NVFP4_OBJ_MSE
    block = wl.block
    xd = [x.to(DEV) for _, x, _ in ts]
    wd = [w.to(DEV) for _, _, w in ts] if wmse else None
    st = ST.for_workload(wl, xd, wd)
    st()
    torch.cuda.synchronize()
    assert st.status.item() == 0
    blocks = ties = 0
    for i, (t, x, w) in enumerate(ts):
        xs = x.float().numpy()
        So, bad = oracle.global_scale(xs, wl.fp8_div)
        assert st.S[i].item() == np.float32(So) and not bad, f"{t.name}: S"
        rows, cols = x.shape
        o = st.outs[i]
        wn = w.numpy() if wmse else None
        ref = oracle.quantize(0, xs, block, So, obj, w=wn, w_row_stride=0, nthreads=_threads())
        gpu = {"codes": o["codes"].cpu(), "sf_linear": o["sf_linear"].cpu(),
               "sf_swizzled": o["sf_swizzled"].cpu() if o["sf_swizzled"] is not None else None}
        stats = compare_quantize(xs, So, block, obj, w if wmse else None, 0, gpu, ref)
        blocks += stats["blocks"]
        ties += stats["near_tie_accepted"]

        # dequantisation of the GPU's codes: bit-exact against the oracle's
        deq = torch.empty(rows, cols, device=DEV)
        if o["sf_swizzled"] is not None:
            B.nvfp4_dequantize(o["codes"], o["sf_swizzled"], B.NVFP4_SF_SWIZZLED, st.S[i:i + 1], rows, cols, block,
                               deq)
        else:
            B.nvfp4_dequantize(o["codes"], o["sf_linear"], B.NVFP4_SF_LINEAR, st.S[i:i + 1], rows, cols, block, deq)
        torch.cuda.synchronize()
        want = oracle.dequantize(gpu["codes"].numpy(), gpu["sf_linear"].numpy(), oracle.LAYOUT_LINEAR, So, rows,
                                 cols, block)
        assert np.array_equal(deq.cpu().numpy().view(np.uint32), want.view(np.uint32)), f"{t.name}: dequant"
        del want

        # summed loss: x-domain loss of the GPU's output vs the oracle's summed block optimum
        err = (xd[i].double() - deq.double()) ** 2
        if wmse:
            err = err * wd[i].double()
        tot_gpu = float(err.sum())
        bl = ref["best"].copy()
        if stats["near_tie_accepted"]:
            d = np.nonzero(gpu["sf_linear"].numpy().reshape(-1) != ref["sf"].reshape(-1))[0]
            bl[d] = oracle.block_losses_at(xs, block, So, gpu["sf_linear"].numpy(), obj, w=wn, w_row_stride=0,
                                           nthreads=_threads())[d]
        tot_ref = float(bl.sum()) * float(So) ** 2
        assert abs(tot_gpu - tot_ref) <= 1e-5 * tot_ref, f"{t.name}: summed loss {tot_gpu} vs {tot_ref}"
        del deq, err, ref
    with capsys.disabled():
        print(f"\n[parity] {name}: {blocks} blocks checked against the oracle, {ties} near-ties accepted")
    del st, xd, wd
    torch.cuda.empty_cache()
