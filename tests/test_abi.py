"""The C-ABI library builds, loads and exports every entry point declared in
include/nvfp4ss.h; argument validation happens on the host before any CUDA
call, so it is exercised here without a GPU (no compute call is made)."""
import ctypes
import os
import re

import pytest

from conftest import ROOT

HEADER = os.path.join(ROOT, "include", "nvfp4ss.h")


def declared_functions():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\**\s+([a-z0-9_]+)\s*\(", src, re.M)))


@pytest.fixture(scope="module")
def L():
    from paper_2606_07618_gb300 import binding
    return binding.lib()


def test_header_declares_the_api():
    assert declared_functions() == sorted([
        "nvfp4_status_string", "nvfp4_global_scale_workspace", "nvfp4_global_scale", "nvfp4_global_scale_noalloc",
        "scalesweep_quantize", "absmax_quantize", "four_over_six_quantize", "nvfp4_dequantize",
        "nvfp4_dynamic_workspace", "scalesweep_quantize_dynamic", "absmax_quantize_dynamic",
        "nvfp4_optimal_scale", "nvfp4_ldlq_prepare_workspace", "nvfp4_ldlq_prepare", "nvfp4_ldlq_workspace",
        "ldlq_quantize", "scalesweep_quantize_group_workspace", "scalesweep_quantize_group",
        "scalesweep_quantize_group_scheduled", "absmax_quantize_group", "nvfp4_selftest_wait_timeout", "nvfp4_row_shard_layout"])


def test_library_exports_every_declared_symbol(L):
    for name in declared_functions():
        assert hasattr(L, name), name


def test_status_strings(L):
    from paper_2606_07618_gb300 import binding
    assert binding.nvfp4_status_string(0) == "ok"
    assert binding.nvfp4_status_string(3) == "misaligned pointer"
    assert binding.nvfp4_global_scale_workspace(1 << 30) >= 8


FAKE = 0x10000000  # never dereferenced: every call below fails validation first


def _ss(L, x=FAKE, dt=0, rows=4, cols=64, block=16, S=FAKE, obj=0, w=None, stride=0, lo=-(2 ** 31), hi=-(2 ** 31),
        codes=FAKE + 0x100000, sfl=FAKE + 0x200000, sfs=None, loss=None):
    return L.scalesweep_quantize(x, dt, rows, cols, block, S, obj, w, stride, lo, hi, codes, sfl, sfs, loss, None)


def test_validation_without_gpu(L):
    assert _ss(L, block=8) == 2                       # unsupported block
    assert _ss(L, block=32, sfs=FAKE + 0x300000) == 2  # swizzled needs block 16
    assert _ss(L, cols=40) == 1                       # cols % block
    assert _ss(L, rows=-1) == 1
    assert _ss(L, dt=7) == 1
    assert _ss(L, obj=3) == 1
    assert _ss(L, lo=-3, hi=-4) == 1                  # empty window
    assert _ss(L, lo=-127, hi=7) == 1
    assert _ss(L, lo=-(2 ** 31), hi=7) == 1           # half-default window
    assert _ss(L, rows=0) == 0                        # empty input: nothing to do, no launch
    assert _ss(L, x=None) == 1
    assert _ss(L, sfl=None) == 1                      # no scale output at all
    assert _ss(L, obj=1, w=None) == 1                 # WMSE needs weights
    assert _ss(L, obj=1, w=FAKE + 0x400000, stride=8) == 1  # stride shorter than a row
    assert _ss(L, x=FAKE + 2) == 3                    # misaligned input
    assert _ss(L, codes=FAKE + 0x100004) == 3         # misaligned codes
    assert _ss(L, obj=1, w=FAKE + 0x400004) == 3      # misaligned weights
    assert _ss(L, codes=FAKE) == 1                    # output overlaps input
    assert _ss(L, sfl=FAKE + 0x100010) == 1           # outputs overlap each other
    assert _ss(L, rows=2 ** 40, cols=2 ** 40) == 4    # size overflow
    assert L.nvfp4_global_scale(FAKE, 0, 100, ctypes.c_float(0.0), FAKE + 4096, None, FAKE + 8192, 1 << 20, None) == 1
    assert L.nvfp4_global_scale(FAKE + 2, 0, 100, ctypes.c_float(256.0), FAKE + 4096, None, FAKE + 8192, 1 << 20,
                                None) == 3
    assert L.nvfp4_global_scale(FAKE, 0, 100, ctypes.c_float(256.0), FAKE + 4096, None, FAKE + 8192, 16, None) == 1
    # the allocation-free global scale refuses inputs past its static scratch
    # (2^29 bf16 / 2^28 fp32 elements) on the host, before any CUDA call
    for dt, n in ((0, (1 << 29) + 1), (1, (1 << 28) + 1)):
        assert L.nvfp4_global_scale_noalloc(FAKE, dt, n, ctypes.c_float(256.0), FAKE + 4096, None, None) == 4
    assert L.nvfp4_global_scale_noalloc(FAKE + 2, 0, 100, ctypes.c_float(256.0), FAKE + 4096, None, None) == 3
    assert L.nvfp4_global_scale_noalloc(FAKE, 0, 100, ctypes.c_float(0.0), FAKE + 4096, None, None) == 1
    assert L.nvfp4_dequantize(FAKE, FAKE + 4096, 2, FAKE + 8192, 4, 64, 32, FAKE + 16384, 1, None) == 2
    assert L.nvfp4_dequantize(FAKE, FAKE + 4096, 3, FAKE + 8192, 4, 64, 16, FAKE + 16384, 1, None) == 1
    assert L.nvfp4_dequantize(FAKE, FAKE + 4096, 1, FAKE + 8192, 4, 64, 16, FAKE + 8, 1, None) == 3


def test_ldlq_validation_without_gpu(L):
    f = ctypes.c_float
    ws = 1 << 24
    prep = lambda H=FAKE, n=64, damp=0.01, perm=FAKE + 0x100000, U=FAKE + 0x200000, D=FAKE + 0x300000, \
        wsp=FAKE + 0x400000, wsb=ws: L.nvfp4_ldlq_prepare(H, n, f(damp), perm, U, D, None, wsp, wsb, None)
    assert prep(n=-1) == 1
    assert prep(damp=-1.0) == 1
    assert prep(damp=float("nan")) == 1
    assert prep(n=0) == 0                             # nothing to do, no launch
    assert prep(n=(1 << 20) + 1) == 4
    assert prep(U=None) == 1
    assert prep(wsb=16) == 1                          # workspace too small
    assert prep(H=FAKE + 2) == 3
    assert prep(U=FAKE + 0x8000) == 1                 # U overlaps H (64*64*4 bytes)
    assert L.nvfp4_ldlq_prepare_workspace(4096) >= 4096 * 4
    assert L.nvfp4_ldlq_workspace(4096, 4096) >= 4096 * 4096 * 5
    assert L.nvfp4_ldlq_workspace(-1, 64) == 0
    q = lambda W=FAKE, dt=0, rows=4, cols=64, block=16, S=FAKE + 0x100000, sf=FAKE + 0x110000, \
        perm=FAKE + 0x120000, U=FAKE + 0x130000, codes=FAKE + 0x200000, wsp=FAKE + 0x400000, wsb=ws: \
        L.ldlq_quantize(W, dt, rows, cols, block, S, sf, perm, U, codes, None, wsp, wsb, None)
    assert q(block=8) == 2
    assert q(cols=40) == 1
    assert q(dt=5) == 1
    assert q(rows=0) == 0
    assert q(perm=None) == 1
    assert q(wsb=64) == 1
    assert q(W=FAKE + 1) == 3
    assert q(codes=FAKE) == 1                         # codes overlap W
    assert q(wsp=FAKE + 0x130000) == 1                # workspace overlaps U



def test_group_validation_without_gpu(L):
    """Argument checks of scalesweep_quantize_group / absmax_quantize_group that return before any CUDA
    call (the overlap checks, which need device pointers to pass, are
    exercised with real buffers in the GPU tests)."""
    from paper_2606_07618_gb300 import binding as B
    f = ctypes.c_float

    def desc(first=None, every=None):
        arr = (B.GroupTensor * 2)()
        for i in range(2):
            t = dict(x=FAKE + i * 0x100000, rows=4, cols=64, w=None, w_row_stride=0,
                     codes=FAKE + 0x1000000 + i * 0x100000, sf_linear=FAKE + 0x2000000 + i * 0x100000,
                     sf_swizzled=None)
            t.update(every or {})
            if i == 0:
                t.update(first or {})
            arr[i] = B.GroupTensor(**t)
        return arr

    S, st, ws = FAKE + 0x3000000, FAKE + 0x3000100, FAKE + 0x3001000
    g = lambda d, n=2, dt=0, obj=0, div=256.0, S=S, ws=ws, wsb=256, block=16: \
        L.scalesweep_quantize_group(d, n, dt, block, obj, f(div), S, st, ws, wsb, None)
    a = lambda d, n=2, dt=0, div=256.0, S=S, ws=ws, wsb=256, block=16: \
        L.absmax_quantize_group(d, n, dt, block, f(div), S, st, ws, wsb, None)
    assert L.scalesweep_quantize_group_workspace() >= 128
    assert g(desc(), n=0) == 1                        # empty group
    assert g(desc(), n=17) == 1                       # more than NVFP4_GROUP_MAX
    assert g(desc(), dt=3) == 1
    assert g(desc(), obj=2) == 1
    assert g(desc(), div=-1.0) == 1
    assert g(desc(), S=None) == 1
    assert g(desc(), ws=None) == 1                    # dynamic scales need the workspace
    assert g(desc(), wsb=16) == 1
    assert g(desc(), ws=FAKE + 0x3001004) == 3
    assert g(desc(), S=S + 2) == 3
    assert g(desc({"cols": 40})) == 1                 # cols % 16
    assert g(desc({"x": FAKE + 2})) == 3
    assert g(desc({"codes": FAKE + 0x1000004})) == 3
    assert g(desc({"sf_linear": None})) == 1          # no scale output
    assert g(desc(), obj=1) == 1                      # WMSE needs weights
    assert g(desc(every={"w": FAKE + 0x4000004}), obj=1) == 3
    assert g(desc(every={"w": FAKE + 0x4000000, "w_row_stride": 8}), obj=1) == 1
    assert g(desc({"rows": 2 ** 40, "cols": 2 ** 40})) == 4
    assert g(desc(), block=8) == 2                    # block not in {16, 32, 64}
    assert g(desc({"cols": 48}), block=32) == 1       # cols % block
    assert g(desc({"sf_swizzled": FAKE + 0x5000000}), block=32) == 2   # swizzled scales need block 16
    sch = lambda d, schedule, n=2: L.scalesweep_quantize_group_scheduled(d, n, 0, 16, 0, f(256.0), S, st, ws, 256,
                                                                          schedule, None)
    assert sch(desc(), 3) == 1                        # unknown schedule
    assert sch(desc(), -1) == 1
    assert sch(desc(), 2, n=0) == 1                   # the other checks apply under every schedule
    assert sch(desc({"x": FAKE + 2}), 2) == 3
    assert a(desc(), n=0) == 1
    assert a(desc(), block=128) == 2
    assert a(desc(), ws=None) == 1
    assert a(desc({"x": FAKE + 2})) == 3
    assert a(desc({"sf_swizzled": FAKE + 0x5000000}), block=64) == 2
    st_test = lambda which=0, status=st, rows=4: L.nvfp4_selftest_wait_timeout(
        which, FAKE, rows, 64, S, status, ws, 1 << 12, FAKE + 0x1000000, FAKE + 0x2000000, None)
    assert st_test(which=2) == 1
    assert st_test(status=None) == 1                 # the status word is how the timeout is seen
    assert st_test(rows=0) == 1


def test_header_constants_and_struct_layout_match_the_binding(tmp_path):
    """Compile a C probe against include/nvfp4ss.h with the host C compiler and
    compare the enum values, the window and group constants and the layouts of
    nvfp4_group_tensor and nvfp4_row_shard with what the Python binding passes
    through ctypes."""
    import shutil
    import subprocess
    from paper_2606_07618_gb300 import binding as B
    cc = shutil.which("gcc") or shutil.which("cc")
    if cc is None:
        pytest.skip("no host C compiler")
    src = tmp_path / "probe.c"
    src.write_text(r'''
#include <stdio.h>
#include "nvfp4ss.h"
#define F(name) printf(#name " %zu %zu\n", offsetof(nvfp4_group_tensor, name), sizeof(((nvfp4_group_tensor*)0)->name))
#define R(name) printf("shard_" #name " %zu %zu\n", offsetof(nvfp4_row_shard, name), sizeof(((nvfp4_row_shard*)0)->name))
int main(void) {
    printf("size %zu\n", sizeof(nvfp4_group_tensor));
    F(x); F(rows); F(cols); F(w); F(w_row_stride); F(codes); F(sf_linear); F(sf_swizzled);
    printf("shard_size %zu\n", sizeof(nvfp4_row_shard));
    R(row_begin); R(row_end); R(x_offset); R(codes_offset); R(sf_linear_offset); R(sf_swizzled_offset);
    R(sf_swizzled_bytes);
    printf("NVFP4_IN_BF16 %d\nNVFP4_IN_F32 %d\nNVFP4_OBJ_MSE %d\nNVFP4_OBJ_WMSE %d\n", NVFP4_IN_BF16, NVFP4_IN_F32,
           NVFP4_OBJ_MSE, NVFP4_OBJ_WMSE);
    printf("NVFP4_SF_LINEAR %d\nNVFP4_SF_SWIZZLED %d\n", NVFP4_SF_LINEAR, NVFP4_SF_SWIZZLED);
    printf("NVFP4_WINDOW_DEFAULT %d\nNVFP4_WINDOW_TIGHT %d\nNVFP4_GROUP_MAX %d\n", NVFP4_WINDOW_DEFAULT,
           NVFP4_WINDOW_TIGHT, NVFP4_GROUP_MAX);
    printf("NVFP4_GROUP_SCHEDULE_AUTO %d\nNVFP4_GROUP_SCHEDULE_TWO_PHASE %d\nNVFP4_GROUP_SCHEDULE_PIPELINED %d\n",
           NVFP4_GROUP_SCHEDULE_AUTO, NVFP4_GROUP_SCHEDULE_TWO_PHASE, NVFP4_GROUP_SCHEDULE_PIPELINED);
    return 0;
}
''')
    exe = tmp_path / "probe"
    subprocess.run([cc, "-std=c99", "-I", os.path.dirname(HEADER), str(src), "-o", str(exe)], check=True)
    out = subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split("\n")
    vals = {ln.split()[0]: [int(v) for v in ln.split()[1:]] for ln in out if ln.strip()}
    assert vals["size"] == [ctypes.sizeof(B.GroupTensor)]
    for name, _ in B.GroupTensor._fields_:
        f = getattr(B.GroupTensor, name)
        assert vals[name] == [f.offset, f.size], name
    assert vals["shard_size"] == [ctypes.sizeof(B.RowShard)]
    for name, _ in B.RowShard._fields_:
        f = getattr(B.RowShard, name)
        assert vals["shard_" + name] == [f.offset, f.size], name
    for name in ("NVFP4_IN_BF16", "NVFP4_IN_F32", "NVFP4_OBJ_MSE", "NVFP4_OBJ_WMSE", "NVFP4_SF_LINEAR",
                 "NVFP4_SF_SWIZZLED", "NVFP4_WINDOW_DEFAULT", "NVFP4_WINDOW_TIGHT", "NVFP4_GROUP_MAX",
                 "NVFP4_GROUP_SCHEDULE_AUTO", "NVFP4_GROUP_SCHEDULE_TWO_PHASE", "NVFP4_GROUP_SCHEDULE_PIPELINED"):
        assert vals[name] == [getattr(B, name)], name


def _declared_signatures():
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    sigs = {}
    for m in re.finditer(r"^\s*(?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\**\s+([a-z0-9_]+)\s*\(([^)]*)\)\s*;", src, re.M):
        params = [p.strip() for p in m.group(2).replace("\n", " ").split(",") if p.strip()]
        if params == ["void"]:
            params = []
        sigs[m.group(1)] = params
    return sigs


def _ctype_of(param):
    from paper_2606_07618_gb300 import binding as B
    decl = param.rsplit(None, 1)[0] if not param.endswith("*") else param
    if "*" in param:
        if "nvfp4_group_tensor" in param:
            return ctypes.POINTER(B.GroupTensor)
        if "nvfp4_row_shard" in param:
            return ctypes.POINTER(B.RowShard)
        return ctypes.c_void_p
    t = decl.replace("const", "").strip()
    return {"int": ctypes.c_int, "int64_t": ctypes.c_int64, "float": ctypes.c_float, "size_t": ctypes.c_size_t,
            "nvfp4_dtype": ctypes.c_int, "nvfp4_objective": ctypes.c_int, "nvfp4_sf_layout": ctypes.c_int,
            "nvfp4_group_schedule": ctypes.c_int, "nvfp4_status": ctypes.c_int}[t]


def _declared_return_types():
    src = re.sub(r"/\*.*?\*/", "", open(HEADER).read(), flags=re.S)
    return {m.group(2): m.group(1).strip() for m in
            re.finditer(r"^\s*((?:const\s+)?[A-Za-z_][A-Za-z0-9_]*\s*\**)\s+([a-z0-9_]+)\s*\(", src, re.M)}


def test_binding_argtypes_match_the_header(L):
    """Every entry point's ctypes argument list has the header's arity and C types
    (pointers as void*, enums as int), so no argument is passed at the wrong width,
    and its result type is the header's (status as int, sizes as size_t)."""
    sigs = _declared_signatures()
    assert sorted(sigs) == declared_functions()
    ret = {"nvfp4_status": ctypes.c_int, "size_t": ctypes.c_size_t, "const char*": ctypes.c_char_p}
    for name, rt in _declared_return_types().items():
        assert getattr(L, name).restype == ret[rt.replace(" *", "*")], (name, rt)
    for name, params in sigs.items():
        got = getattr(L, name).argtypes
        assert got is not None, name
        want = [_ctype_of(p) for p in params]
        assert len(got) == len(want), name
        for i, (g, w) in enumerate(zip(got, want)):
            assert g == w, (name, i, params[i])


def test_build_covers_every_source_for_sm_103a():
    """Every CUDA translation unit in csrc/ is compiled, for sm_103a only, and
    every header it includes counts towards the rebuild check."""
    from paper_2606_07618_gb300 import build as Bd
    cu = sorted(f for f in os.listdir(Bd.CSRC) if f.endswith(".cu"))
    assert sorted(Bd.SOURCES) == cu
    assert Bd.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
    flags = Bd._flags(False)
    assert "-O3" in flags and "-lineinfo" in flags
    inputs = set(os.path.basename(f) for f in Bd._inputs())
    headers = {f for f in os.listdir(Bd.CSRC) if f.endswith((".h", ".cuh"))} | {"nvfp4ss.h"}
    assert headers | set(cu) <= inputs
