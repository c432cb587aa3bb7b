"""nvfp4_global_scale_noalloc: the global-scale entry point for callers that
cannot allocate device memory (a fixed device-memory plan, or a host without an
allocator of its own), which keeps its scratch in a static device array.

Called through the C ABI, it must give the same S and status word as
nvfp4_global_scale with a caller-provided workspace, on two calls in a row
(the second call reuses the scratch the first one left behind), and the same S
as the CPU oracle.  Its refusal of inputs larger than the scratch covers is a
host-side check, tested without a GPU in test_abi.py.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle

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


def with_workspace(B, x, D):
    S = torch.empty(1, dtype=torch.float32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    ws = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
    B.nvfp4_global_scale(x, D, S, st, ws)
    return S, st


def without_workspace(B, x, D):
    S = torch.full((1,), -1.0, dtype=torch.float32, device=DEV)
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    L = B.lib()
    rc = L.nvfp4_global_scale_noalloc(ctypes.c_void_p(x.data_ptr()), B.NVFP4_IN_BF16 if x.dtype == torch.bfloat16
                                      else B.NVFP4_IN_F32, x.numel(), ctypes.c_float(D),
                                      ctypes.c_void_p(S.data_ptr()), ctypes.c_void_p(st.data_ptr()),
                                      ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))
    assert rc == 0, B.nvfp4_status_string(rc)
    return S, st


@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_no_alloc_global_scale_matches_workspace_version(B, dtype):
    g = torch.Generator().manual_seed(17)
    a = (torch.randn(3 * 1024 * 1024 + 5, generator=g) * 2.5).to(dtype).to(DEV)   # large input first
    b = (torch.randn(1000, generator=g) * 0.01).to(dtype).to(DEV)                  # then a small one
    b[17] = float("inf")
    for x, D, flagged in ((a, 256.0, 0), (b, 448.0, 1)):
        S0, st0 = with_workspace(B, x, D)
        S1, st1 = without_workspace(B, x, D)
        torch.cuda.synchronize()
        assert S1.item() == S0.item() or (np.isinf(S1.item()) and np.isinf(S0.item()))
        assert st1.item() == st0.item() == flagged
        So, bad = oracle.global_scale(x.float().cpu().numpy(), D)
        assert S1.item() == np.float32(So) and bad == bool(flagged)
