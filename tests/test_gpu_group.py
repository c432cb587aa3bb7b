"""Grouped ScaleSweep launch (scalesweep_quantize_group) on the GPU.

One launch quantises a list of tensors and, with a dynamic global scale,
reduces each tensor's amax inside the same launch.  For every tensor it must
give the oracle's codes and scales (near-tie rule of parity.py) and, bit for
bit, what the per-tensor entry points give: nvfp4_global_scale then
scalesweep_quantize (S, codes, linear and swizzled scales).  Shapes are
ragged on purpose: segment counts that are not multiples of 32 (a warp), rows
not multiples of 128 and scale columns not multiples of 4 (swizzle pads), a
one-row tensor, an empty tensor, an all-zero tensor.
"""
import numpy as np
import pytest
import torch

import oracle
from parity import compare_quantize
from paper_2606_07618_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"
WIN = None


@pytest.fixture(scope="module")
def B():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2606_07618_gb300 import binding
    binding.lib()
    oracle.build()
    global WIN
    WIN = (binding.NVFP4_WINDOW_DEFAULT, binding.NVFP4_WINDOW_DEFAULT)
    return binding


SHAPES = [(130, 192), (1, 64), (37, 48), (300, 512), (0, 64), (2048, 1024), (64, 80)]


def make_group(dtype, obj, seed=0, shapes=SHAPES, row_weights=(3,)):
    xs, ws, strides = [], [], []
    for i, (r, c) in enumerate(shapes):
        if r == 0:
            x = torch.empty(0, c, dtype=torch.bfloat16)
        else:
            x = W.small_tensor(r, c, 100 * seed + i, dist="student_t" if i % 2 else "normal", std=0.02 + 0.01 * i,
                               outliers=1 + i % 3, mult=20.0 + i)
        if i == 6 and r > 0:
            x = torch.zeros(r, c, dtype=torch.bfloat16)          # an all-zero tensor: S = 0, signs only
        xs.append(x.to(dtype))
        if obj == 1:
            g = torch.Generator().manual_seed(seed * 31 + i)
            if i in row_weights:                                   # per-element weights, padded row stride
                stride = c + 4
                w = torch.exp(torch.randn(max(r, 1), stride, generator=g))
            else:
                stride = 0
                w = torch.exp(torch.randn(c, generator=g))
            ws.append(w)
            strides.append(stride)
        else:
            ws.append(None)
            strides.append(0)
    return xs, ws, strides


def run_group(B, xs, ws, strides, obj, D=256.0, S_in=None, ws_buf=None, status=None, block=16, method=0,
              schedule=None):
    dev_x = [x.to(DEV) for x in xs]
    dev_w = [w.to(DEV) if w is not None else None for w in ws]
    outs = [B.empty_outputs(x.shape[0], x.shape[1], block, device=DEV, linear=True, swizzled=block == 16)
            for x in xs]
    for o in outs:                                                   # poison: every byte must be written
        for k in ("codes", "sf_linear", "sf_swizzled"):
            if o[k] is not None:
                o[k].fill_(0xEE)
    desc = B.group_descriptors(dev_x, dev_w, strides, [o["codes"] for o in outs], [o["sf_linear"] for o in outs],
                               [o["sf_swizzled"] for o in outs])
    dt = B.NVFP4_IN_BF16 if xs[0].dtype == torch.bfloat16 else B.NVFP4_IN_F32
    st = status if status is not None else torch.zeros(1, dtype=torch.int32, device=DEV)
    call = (lambda d, S_, ws_: B.scalesweep_quantize_group(desc, dt, obj, d, S_, st, ws_, block=block,
                                                           schedule=schedule)) \
        if method == 0 else (lambda d, S_, ws_: B.absmax_quantize_group(desc, dt, d, S_, st, ws_, block=block))
    if S_in is None:
        S = torch.full((len(xs),), -1.0, device=DEV)
        if ws_buf is None:
            ws_buf = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
        call(D, S, ws_buf)
    else:
        S = S_in.clone()
        call(0.0, S, None)
    torch.cuda.synchronize()
    return S, st, outs, dev_x, dev_w


def per_tensor(B, x, w, stride, obj, S=None, D=256.0, block=16, method=0):
    st = torch.zeros(1, dtype=torch.int32, device=DEV)
    if S is None:
        S = torch.empty(1, device=DEV)
        wsb = torch.empty(B.nvfp4_global_scale_workspace(x.numel()), dtype=torch.uint8, device=DEV)
        B.nvfp4_global_scale(x, D, S, st, wsb)
    o = B.empty_outputs(x.shape[0], x.shape[1], block, device=DEV, linear=True, swizzled=block == 16)
    if x.numel():
        if method == 0:
            B.scalesweep_quantize(x, block, S, obj, w, stride, *WIN, o["codes"], o["sf_linear"], o["sf_swizzled"],
                                  None)
        else:
            B.absmax_quantize(x, block, S, o["codes"], o["sf_linear"], o["sf_swizzled"], None)
    torch.cuda.synchronize()
    return S, st, o


def check_against_per_tensor(B, xs, ws, strides, obj, S, outs, dev_x, dev_w, static=False, block=16, method=0):
    for i, x in enumerate(dev_x):
        S1, _, o1 = per_tensor(B, x, dev_w[i], strides[i], obj, S=S[i:i + 1] if static else None, block=block,
                               method=method)
        if not static:
            assert S[i].item() == S1.item(), f"tensor {i}: S {S[i].item()} vs {S1.item()}"
        if x.numel() == 0:
            continue
        for k in ("codes", "sf_linear", "sf_swizzled"):
            if o1[k] is not None:
                assert torch.equal(outs[i][k], o1[k]), f"tensor {i}: {k}"


SCHEDULES = [None, 1, 2]        # the library's choice, two-phase, pipelined


@pytest.mark.parametrize("schedule", SCHEDULES)
@pytest.mark.parametrize("obj", [0, 1])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_group_dynamic_matches_oracle_and_per_tensor(B, dtype, obj, schedule):
    xs, ws, strides = make_group(dtype, obj, seed=1)
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, obj, schedule=schedule)
    assert st.item() == 0
    check_against_per_tensor(B, xs, ws, strides, obj, S, outs, dev_x, dev_w)
    for i, x in enumerate(xs):
        xs_np = x.float().numpy()
        So, bad = oracle.global_scale(xs_np, 256.0) if x.numel() else (0.0, False)
        assert S[i].item() == np.float32(So), f"tensor {i}"
        if x.numel() == 0:
            continue
        wn = ws[i].numpy() if ws[i] is not None else None
        ref = oracle.quantize(0, xs_np, 16, So, obj, w=wn, w_row_stride=strides[i])
        compare_quantize(xs_np, So, 16, obj, ws[i], strides[i], outs[i], ref)


SHAPES64 = [(130, 192), (1, 64), (37, 128), (300, 512), (0, 64), (1000, 1024), (64, 320)]


@pytest.mark.parametrize("dyn", [True, False, "pipelined"])
@pytest.mark.parametrize("block,obj,method", [(32, 0, 0), (32, 1, 0), (64, 0, 0), (64, 1, 0),
                                              (16, 0, 1), (32, 0, 1), (64, 0, 1)])
@pytest.mark.parametrize("dtype", [torch.bfloat16, torch.float32])
def test_group_blocks_and_absmax(B, dtype, block, obj, method, dyn):
    """Blocks of 32 and 64 (two and four lanes per block) and the grouped AbsMax
    launch: every tensor equals the oracle (near-tie rule) and, bit for bit,
    the per-tensor call with the same scale.  "pipelined": dynamic scales under
    the pipelined schedule (AbsMax has no such schedule)."""
    if dyn == "pipelined" and method == 1:
        pytest.skip("the pipelined schedule is a ScaleSweep schedule")
    xs, ws, strides = make_group(dtype, obj, seed=7 + block + 3 * method, shapes=SHAPES64)
    S_in = None
    if not dyn:
        S_in = torch.tensor([oracle.global_scale(x.float().numpy(), 256.0)[0] if x.numel() else 1.0 for x in xs],
                            dtype=torch.float32, device=DEV)
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, obj, S_in=S_in, block=block, method=method,
                                          schedule=2 if dyn == "pipelined" else None)
    assert st.item() == 0
    check_against_per_tensor(B, xs, ws, strides, obj, S, outs, dev_x, dev_w, static=not dyn, block=block,
                             method=method)
    for i, x in enumerate(xs):
        if x.numel() == 0:
            continue
        xs_np = x.float().numpy()
        So = float(S[i].item())
        if dyn:
            assert So == np.float32(oracle.global_scale(xs_np, 256.0)[0]), f"tensor {i}"
        wn = ws[i].numpy() if ws[i] is not None else None
        ref = oracle.quantize(method, xs_np, block, So, obj if method == 0 else 0, w=wn if method == 0 else None,
                              w_row_stride=strides[i])
        compare_quantize(xs_np, So, block, obj, ws[i], strides[i], outs[i], ref, method=method)


@pytest.mark.parametrize("obj", [0, 1])
def test_group_static_scales(B, obj):
    xs, ws, strides = make_group(torch.bfloat16, obj, seed=2)
    S_in = torch.tensor([oracle.global_scale(x.float().numpy(), 448.0)[0] if x.numel() else 1.0 for x in xs],
                        dtype=torch.float32, device=DEV)
    S_in[2] = 0.0                                                  # a zero scale: signs only
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, obj, S_in=S_in)
    assert torch.equal(S, S_in) and st.item() == 0
    check_against_per_tensor(B, xs, ws, strides, obj, S, outs, dev_x, dev_w, static=True)


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_group_single_tensor_and_many_tensors(B, schedule):
    # one tensor; and the maximum of 16 tensors of assorted small shapes
    xs, ws, strides = make_group(torch.bfloat16, 1, seed=3, shapes=[(513, 4096)], row_weights=())
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, 1, schedule=schedule)
    check_against_per_tensor(B, xs, ws, strides, 1, S, outs, dev_x, dev_w)
    shapes = [(1 + 37 * i, 16 * (1 + (5 * i) % 23)) for i in range(16)]
    xs, ws, strides = make_group(torch.bfloat16, 0, seed=4, shapes=shapes)
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, 0, schedule=schedule)
    assert st.item() == 0
    check_against_per_tensor(B, xs, ws, strides, 0, S, outs, dev_x, dev_w)


@pytest.mark.parametrize("obj", [0, 1])
def test_group_schedules_agree_on_large_tensors(B, obj):
    """Tensors large enough that the pipelined schedule's reduction of the
    smaller ones runs beside the largest one's sweep (bf16, 117M elements in
    three tensors): S, codes and both scale layouts are the same bytes under
    both schedules."""
    shapes = [(4096, 4096), (1024, 8192), (12288, 8192)]
    xs = [W.small_tensor(r, c, 60 + i, dist="normal", std=0.02, outliers=4, mult=20.0) for i, (r, c) in
          enumerate(shapes)]
    ws = [torch.exp(torch.randn(c, generator=torch.Generator().manual_seed(70 + i))) if obj else None
          for i, (_, c) in enumerate(shapes)]
    res = [run_group(B, xs, ws, [0] * 3, obj, schedule=sch) for sch in (1, 2)]
    (S1, st1, o1, _, _), (S2, st2, o2, _, _) = res
    assert st1.item() == 0 and st2.item() == 0 and torch.equal(S1, S2)
    for i, (xn, Si) in enumerate(zip(xs, S1.tolist())):
        assert Si == np.float32(oracle.global_scale(xn.float().numpy(), 256.0)[0])
        for k in ("codes", "sf_linear", "sf_swizzled"):
            assert torch.equal(o1[i][k], o2[i][k]), (i, k)


def test_group_llama_layer_full_size(B):
    """The Llama-3-8B layer (7 weights, 218M elements, WMSE with lognormal
    channel weights, dynamic S, D = 256) in one launch: every tensor equals the
    per-tensor path bit for bit; S and 24 sampled rows per tensor equal the
    oracle."""
    wl = W.workload("llama8b")
    xs = [W.draw(t) for t in wl.tensors]
    ws = [W.draw_weights(t) for t in wl.tensors]
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, [0] * len(xs), 1, D=wl.fp8_div)
    assert st.item() == 0
    check_against_per_tensor(B, xs, ws, [0] * len(xs), 1, S, outs, dev_x, dev_w)
    for i, (t, x) in enumerate(zip(wl.tensors, xs)):
        xs_np = x.float().numpy()
        So, _ = oracle.global_scale(xs_np, wl.fp8_div)
        assert S[i].item() == np.float32(So), t.name
        idx = np.unique(np.linspace(0, t.rows - 1, 24).astype(np.int64))
        sub = {"codes": outs[i]["codes"][idx], "sf_linear": outs[i]["sf_linear"][idx]}
        ref = oracle.quantize(0, xs_np[idx], 16, So, 1, w=ws[i].numpy())
        compare_quantize(xs_np[idx], So, 16, 1, ws[i], 0, sub, ref)


@pytest.mark.parametrize("schedule", SCHEDULES)
def test_group_nonfinite_flag_reuse_and_empty(B, schedule):
    xs, ws, strides = make_group(torch.bfloat16, 0, seed=5)
    wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
    ref = None
    for _ in range(3):                                             # one workspace, back to back
        S, st, outs, _, _ = run_group(B, xs, ws, strides, 0, ws_buf=wsb, schedule=schedule)
        assert st.item() == 0
        if ref is None:
            ref = (S.clone(), outs)
        else:
            assert torch.equal(S, ref[0])
            for a, b in zip(outs, ref[1]):
                for k in ("codes", "sf_linear", "sf_swizzled"):
                    assert torch.equal(a[k], b[k])
    bad = [x.clone() for x in xs]
    bad[3][5, 7] = float("inf")
    S, st, _, _, _ = run_group(B, bad, ws, strides, 0, ws_buf=wsb, schedule=schedule)
    assert st.item() == 1
    assert S[3].item() == float("inf") and torch.equal(S[:3], ref[0][:3])
    bad = [x.clone() for x in xs]
    bad[5][0, 0] = float("nan")
    S, st, _, _, _ = run_group(B, bad, ws, strides, 0, ws_buf=wsb, schedule=schedule)
    assert st.item() == 1 and S[5].item() == ref[0][5].item()        # NaN is skipped by the max
    empty = [torch.empty(0, 64, dtype=torch.bfloat16), torch.empty(3, 0, dtype=torch.bfloat16)]
    S, st, _, _, _ = run_group(B, empty, [None, None], [0, 0], 0, ws_buf=wsb, schedule=schedule)
    assert S.tolist() == [0.0, 0.0] and st.item() == 0


def test_group_rejects_overlapping_buffers(B):
    x = torch.zeros(64, 64, dtype=torch.bfloat16, device=DEV)
    codes = torch.empty(64, 32, dtype=torch.uint8, device=DEV)
    sf = torch.empty(64, 4, dtype=torch.uint8, device=DEV)
    S = torch.zeros(2, device=DEV)
    wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
    both = B.group_descriptors([x, x], [None, None], [0, 0], [codes, codes], [sf, None], [None, sf])
    with pytest.raises(B.Nvfp4Error) as e:
        B.scalesweep_quantize_group(both, B.NVFP4_IN_BF16, 0, 256.0, S, None, wsb)
    assert e.value.code == 1
    into_input = B.group_descriptors([x], [None], [0], [x.view(torch.uint8)[:, :32]], [sf], [None])
    with pytest.raises(B.Nvfp4Error) as e:
        B.scalesweep_quantize_group(into_input, B.NVFP4_IN_BF16, 0, 256.0, S, None, wsb)
    assert e.value.code == 1
    ok = B.group_descriptors([x], [None], [0], [codes], [sf], [None])
    B.scalesweep_quantize_group(ok, B.NVFP4_IN_BF16, 0, 256.0, S, None, wsb)
    torch.cuda.synchronize()
    assert S[0].item() == 0.0 and not torch.any(codes & 0x77).item()


def test_group_output_guard_bytes_untouched(B):
    """Outputs of a ragged group carved from one buffer with 4 KiB guards between
    them: every guard byte survives (the 256-segment padding of each tensor's
    range is never written)."""
    shapes = [(37, 48), (130, 192), (1, 64)]
    xs, ws, strides = make_group(torch.bfloat16, 1, seed=7, shapes=shapes, row_weights=())
    G = 4096
    sizes = []
    for r, c in shapes:
        sizes += [r * c // 2, r * c // 16, B.swizzled_bytes(r, c)]
    offs, pos = [], G
    for n in sizes:
        pos = (pos + 15) // 16 * 16
        offs.append(pos)
        pos += n + G
    buf = torch.full((pos,), 0xAB, dtype=torch.uint8, device=DEV)
    views = [buf[o:o + n] for o, n in zip(offs, sizes)]
    codes = [views[3 * i].view(r, c // 2) for i, (r, c) in enumerate(shapes)]
    sfl = [views[3 * i + 1].view(r, c // 16) for i, (r, c) in enumerate(shapes)]
    sfs = [views[3 * i + 2] for i in range(len(shapes))]
    dx = [x.to(DEV) for x in xs]
    dw = [w.to(DEV) for w in ws]
    desc = B.group_descriptors(dx, dw, strides, codes, sfl, sfs)
    S = torch.empty(len(shapes), device=DEV)
    wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
    B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, 1, 256.0, S, None, wsb)
    torch.cuda.synchronize()
    mask = torch.ones(pos, dtype=torch.bool, device=DEV)
    for o, n in zip(offs, sizes):
        mask[o:o + n] = False
    assert torch.all(buf[mask] == 0xAB)
    for i, x in enumerate(dx):
        _, _, o1 = per_tensor(B, x, dw[i], strides[i], 1)
        assert torch.equal(codes[i], o1["codes"]) and torch.equal(sfl[i], o1["sf_linear"])
        assert torch.equal(sfs[i], o1["sf_swizzled"])


@pytest.mark.parametrize("schedule", [1, 2])
def test_group_dynamic_in_cuda_graph(B, schedule):
    """The grouped call (workspace memset, then the cooperative launch or the
    pipelined schedule's four launches) captured in a CUDA graph and replayed
    gives the eager results; the library neither allocates nor synchronises,
    so it can be captured."""
    xs, ws, strides = make_group(torch.bfloat16, 1, seed=8, shapes=[(300, 512), (64, 80), (1024, 256)])
    S, st, outs, dev_x, dev_w = run_group(B, xs, ws, strides, 1, schedule=3 - schedule)
    outs2 = [B.empty_outputs(x.shape[0], x.shape[1], 16, device=DEV, linear=True, swizzled=True) for x in xs]
    desc = B.group_descriptors(dev_x, dev_w, strides, [o["codes"] for o in outs2], [o["sf_linear"] for o in outs2],
                               [o["sf_swizzled"] for o in outs2])
    S2 = torch.zeros(len(xs), device=DEV)
    st2 = torch.zeros(1, dtype=torch.int32, device=DEV)
    wsb = torch.empty(B.scalesweep_quantize_group_workspace(), dtype=torch.uint8, device=DEV)
    g = torch.cuda.CUDAGraph()
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, 1, 256.0, S2, st2, wsb, stream=s,
                                    schedule=schedule)                                         # warm-up
    torch.cuda.synchronize()
    with torch.cuda.graph(g, stream=s):
        B.scalesweep_quantize_group(desc, B.NVFP4_IN_BF16, 1, 256.0, S2, st2, wsb, stream=s, schedule=schedule)
    for _ in range(2):
        for o in outs2:
            o["codes"].zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(S2, S) and st2.item() == 0
        for a, b in zip(outs, outs2):
            for k in ("codes", "sf_linear", "sf_swizzled"):
                assert torch.equal(a[k], b[k])


@pytest.mark.parametrize("activation", [False, True])
def test_zero_copy_host_buffers_equal_device_buffers(B, activation):
    """Inputs and outputs in pinned host memory (the kernels load and store over
    the host link): the same bytes as with device buffers, for the grouped
    launch and for the fused single-tensor launch."""
    from paper_2606_07618_gb300 import step as ST
    shapes = [(300, 512)] if activation else [(300, 512), (130, 192), (64, 1024)]
    xs = [W.small_tensor(r, c, 40 + i, dist="student_t", std=1.0, outliers=2, mult=30.0) for i, (r, c) in
          enumerate(shapes)]
    ws = [torch.exp(torch.randn(c, generator=torch.Generator().manual_seed(i))).to(DEV) for i, (_, c) in
          enumerate(shapes)]
    obj = B.NVFP4_OBJ_WMSE
    dev_step = ST.QuantizeStep([x.to(DEV) for x in xs], ws, objective=obj, activation=activation)
    hx = [x.pin_memory() for x in xs]
    houts = [{k: torch.empty_like(v, device="cpu").pin_memory() if v is not None else None for k, v in o.items()}
             for o in dev_step.outs]
    host_step = ST.QuantizeStep(hx, ws, objective=obj, activation=activation, outs=houts, device=DEV)
    dev_step()
    host_step()
    torch.cuda.synchronize()
    assert torch.equal(dev_step.S, host_step.S) and host_step.status.item() == 0
    for a, b in zip(dev_step.outs, houts):
        for k in ("codes", "sf_linear", "sf_swizzled"):
            assert torch.equal(a[k].cpu(), b[k]), k

