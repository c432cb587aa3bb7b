"""Failure detection on the GPU without a fault: every device wait is bounded.

nvfp4_selftest_wait_timeout raises the arrival target of the dynamic-scale
sweep's grid barrier (which = 0) and of the grouped launch's scale wait
(which = 1) past what the launch can reach.  Each wait must give up after its
limit (about a second), report it in bit 1 of the status word, leave the
outputs unwritten, and leave the context usable: the same call without the
raised target right after gives the normal result.
"""
import time

import pytest
import torch

from paper_2606_07618_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_07618_gb300 import binding
    binding.lib()
    return binding


@pytest.mark.parametrize("which", [0, 1])
def test_wait_runs_out_and_is_reported(B, which):
    x = W.small_tensor(256, 1024, 3).to(DEV)
    ws = torch.empty(max(B.nvfp4_dynamic_workspace(), B.scalesweep_quantize_group_workspace()), dtype=torch.uint8,
                     device=DEV)
    codes = torch.full((256, 512), 0xEE, dtype=torch.uint8, device=DEV)
    sfl = torch.full((256, 64), 0xEE, dtype=torch.uint8, device=DEV)
    S = torch.full((1,), -1.0, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    torch.cuda.synchronize()
    t0 = time.time()
    B.nvfp4_selftest_wait_timeout(which, x, S, st, ws, codes, sfl)
    torch.cuda.synchronize()
    dt = time.time() - t0
    assert st.item() & 2
    assert 0.5 < dt < 60
    assert torch.all(codes == 0xEE) and torch.all(sfl == 0xEE)      # the waiting warps wrote nothing
    # the context is still usable: the real call gives the normal result
    st.zero_()
    win = (B.NVFP4_WINDOW_DEFAULT, B.NVFP4_WINDOW_DEFAULT)
    S2 = torch.empty(1, device=DEV)
    if which == 0:
        B.scalesweep_quantize_dynamic(x, 16, 256.0, 0, None, 0, *win, S2, st, ws, codes, sfl)
    else:
        d = B.group_descriptors([x], [None], [0], [codes], [sfl], [None])
        B.scalesweep_quantize_group(d, B.NVFP4_IN_BF16, 0, 256.0, S2, st, ws)
    ref = B.empty_outputs(256, 1024, 16, device=DEV, linear=True)
    S3 = torch.empty(1, device=DEV)
    gws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, 256.0, S3, None, gws)
    B.scalesweep_quantize(x, 16, S3, 0, None, 0, *win, ref["codes"], ref["sf_linear"])
    torch.cuda.synchronize()
    assert st.item() == 0 and S2.item() == S3.item()
    assert torch.equal(codes, ref["codes"]) and torch.equal(sfl, ref["sf_linear"])
