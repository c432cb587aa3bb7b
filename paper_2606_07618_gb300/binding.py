"""Thin ctypes binding of libnvfp4ss.so (include/nvfp4ss.h).

Every function has the name of the C entry point it calls and only marshals
arguments: torch CUDA tensors become device pointers, the current torch CUDA
stream becomes the cudaStream_t, a non-OK status raises ``Nvfp4Error``.  All
arithmetic runs in the library's CUDA kernels; there is no CPU fallback, and a
missing library raises at load time.
"""
from __future__ import annotations

import ctypes
import os

import torch

from . import build as _build

NVFP4_IN_BF16, NVFP4_IN_F32 = 0, 1
NVFP4_OBJ_MSE, NVFP4_OBJ_WMSE = 0, 1
NVFP4_SF_LINEAR, NVFP4_SF_SWIZZLED = 1, 2
NVFP4_WINDOW_DEFAULT = -(2 ** 31)
NVFP4_WINDOW_TIGHT = -(2 ** 31) + 1

STATUS = {0: "NVFP4_OK", 1: "NVFP4_ERR_INVALID_ARG", 2: "NVFP4_ERR_UNSUPPORTED", 3: "NVFP4_ERR_ALIGNMENT",
          4: "NVFP4_ERR_RANGE", 5: "NVFP4_ERR_CUDA"}


class Nvfp4Error(RuntimeError):
    def __init__(self, fn: str, code: int, msg: str):
        super().__init__(f"{fn}: {STATUS.get(code, code)} ({msg})")
        self.code = code


_lib = None

NVFP4_GROUP_MAX = 16
NVFP4_GROUP_SCHEDULE_AUTO, NVFP4_GROUP_SCHEDULE_TWO_PHASE, NVFP4_GROUP_SCHEDULE_PIPELINED = 0, 1, 2


class RowShard(ctypes.Structure):
    """nvfp4_row_shard: one shard's rows and output offsets (nvfp4_row_shard_layout)."""
    _fields_ = [("row_begin", ctypes.c_int64), ("row_end", ctypes.c_int64), ("x_offset", ctypes.c_int64),
                ("codes_offset", ctypes.c_int64), ("sf_linear_offset", ctypes.c_int64),
                ("sf_swizzled_offset", ctypes.c_int64), ("sf_swizzled_bytes", ctypes.c_int64)]


class GroupTensor(ctypes.Structure):
    """nvfp4_group_tensor: one tensor of a scalesweep_quantize_group call."""
    _fields_ = [("x", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64), ("w", ctypes.c_void_p),
                ("w_row_stride", ctypes.c_int64), ("codes", ctypes.c_void_p), ("sf_linear", ctypes.c_void_p),
                ("sf_swizzled", ctypes.c_void_p)]


def library_path() -> str:
    return _build.LIB


def lib() -> ctypes.CDLL:
    """Load libnvfp4ss.so, building it first if it is missing or stale."""
    global _lib
    if _lib is None:
        if not _build.up_to_date():
            _build.build()
        if not os.path.exists(_build.LIB):
            raise RuntimeError("libnvfp4ss.so is not built and could not be built")
        L = ctypes.CDLL(_build.LIB)
        i, i64, f, p, sz = ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_void_p, ctypes.c_size_t
        L.nvfp4_status_string.argtypes, L.nvfp4_status_string.restype = [i], ctypes.c_char_p
        L.nvfp4_global_scale_workspace.argtypes, L.nvfp4_global_scale_workspace.restype = [i64], sz
        L.nvfp4_global_scale.argtypes = [p, i, i64, f, p, p, p, sz, p]
        L.nvfp4_global_scale_noalloc.argtypes = [p, i, i64, f, p, p, p]
        L.scalesweep_quantize.argtypes = [p, i, i64, i64, i, p, i, p, i64, i, i, p, p, p, p, p]
        L.absmax_quantize.argtypes = [p, i, i64, i64, i, p, p, p, p, p, p]
        L.four_over_six_quantize.argtypes = [p, i, i64, i64, i, p, i, p, i64, p, p, p, p, p]
        L.nvfp4_dequantize.argtypes = [p, p, i, p, i64, i64, i, p, i, p]
        L.nvfp4_dynamic_workspace.argtypes, L.nvfp4_dynamic_workspace.restype = [], sz
        L.scalesweep_quantize_dynamic.argtypes = [p, i, i64, i64, i, f, i, p, i64, i, i, p, p, p, sz, p, p, p, p, p]
        L.absmax_quantize_dynamic.argtypes = [p, i, i64, i64, i, f, p, p, p, sz, p, p, p, p, p]
        L.scalesweep_quantize_group_workspace.argtypes, L.scalesweep_quantize_group_workspace.restype = [], sz
        L.scalesweep_quantize_group.argtypes = [ctypes.POINTER(GroupTensor), i, i, i, i, f, p, p, p, sz, p]
        L.scalesweep_quantize_group_scheduled.argtypes = [ctypes.POINTER(GroupTensor), i, i, i, i, f, p, p, p, sz,
                                                          i, p]
        L.absmax_quantize_group.argtypes = [ctypes.POINTER(GroupTensor), i, i, i, f, p, p, p, sz, p]
        L.nvfp4_selftest_wait_timeout.argtypes = [i, p, i64, i64, p, p, p, sz, p, p, p]
        L.nvfp4_row_shard_layout.argtypes = [i64, i64, i, i, i, ctypes.POINTER(RowShard)]
        L.nvfp4_optimal_scale.argtypes = [p, i, i64, i64, i, p, i, p, i64, p, p, p, p, p]
        L.nvfp4_ldlq_prepare_workspace.argtypes, L.nvfp4_ldlq_prepare_workspace.restype = [i64], sz
        L.nvfp4_ldlq_prepare.argtypes = [p, i64, f, p, p, p, p, p, sz, p]
        L.nvfp4_ldlq_workspace.argtypes, L.nvfp4_ldlq_workspace.restype = [i64, i64], sz
        L.ldlq_quantize.argtypes = [p, i, i64, i64, i, p, p, p, p, p, p, p, sz, p]
        for fn in ("nvfp4_global_scale", "nvfp4_global_scale_noalloc", "scalesweep_quantize", "absmax_quantize",
                   "four_over_six_quantize", "nvfp4_dequantize", "scalesweep_quantize_dynamic",
                   "absmax_quantize_dynamic", "nvfp4_optimal_scale", "nvfp4_ldlq_prepare", "ldlq_quantize",
                   "scalesweep_quantize_group", "scalesweep_quantize_group_scheduled", "absmax_quantize_group",
                   "nvfp4_selftest_wait_timeout",
                   "nvfp4_row_shard_layout"):
            getattr(L, fn).restype = i
        _lib = L
    return _lib


def _ptr(t):
    # plain ints: ctypes converts them for c_void_p parameters without an object
    if t is None or isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _dtype(x) -> int:
    if x.dtype == torch.bfloat16:
        return NVFP4_IN_BF16
    if x.dtype == torch.float32:
        return NVFP4_IN_F32
    raise TypeError(f"unsupported dtype {x.dtype}")


def _check(fn: str, rc: int):
    if rc != 0:
        raise Nvfp4Error(fn, rc, lib().nvfp4_status_string(rc).decode())


def nvfp4_status_string(code: int) -> str:
    return lib().nvfp4_status_string(int(code)).decode()


def nvfp4_global_scale_workspace(n: int) -> int:
    return int(lib().nvfp4_global_scale_workspace(int(n)))


def nvfp4_global_scale(x, fp8_div: float, S_out, status=None, workspace=None, stream=None):
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().nvfp4_global_scale(_ptr(x), _dtype(x), x.numel(), float(fp8_div), _ptr(S_out), _ptr(status),
                                  _ptr(workspace), ws_bytes, _stream(stream))
    _check("nvfp4_global_scale", rc)


def nvfp4_global_scale_noalloc(x, fp8_div: float, S_out, status=None, stream=None):
    """Global scale for callers that cannot allocate: no workspace argument
    (the library's static device scratch is used instead)."""
    rc = lib().nvfp4_global_scale_noalloc(_ptr(x), _dtype(x), x.numel(), float(fp8_div), _ptr(S_out), _ptr(status),
                                          _stream(stream))
    _check("nvfp4_global_scale_noalloc", rc)


def scalesweep_quantize(x, block: int, S, objective: int, w, w_row_stride: int, win_lo: int, win_hi: int,
                        codes, sf_linear=None, sf_swizzled=None, block_loss=None, stream=None):
    rows, cols = x.shape
    rc = lib().scalesweep_quantize(_ptr(x), _dtype(x), rows, cols, int(block), _ptr(S), int(objective), _ptr(w),
                                   int(w_row_stride), int(win_lo), int(win_hi), _ptr(codes), _ptr(sf_linear),
                                   _ptr(sf_swizzled), _ptr(block_loss), _stream(stream))
    _check("scalesweep_quantize", rc)


def absmax_quantize(x, block: int, S, codes, sf_linear=None, sf_swizzled=None, block_loss=None, stream=None):
    rows, cols = x.shape
    rc = lib().absmax_quantize(_ptr(x), _dtype(x), rows, cols, int(block), _ptr(S), _ptr(codes), _ptr(sf_linear),
                               _ptr(sf_swizzled), _ptr(block_loss), _stream(stream))
    _check("absmax_quantize", rc)


def four_over_six_quantize(x, block: int, S, objective: int, w, w_row_stride: int, codes, sf_linear=None,
                           sf_swizzled=None, block_loss=None, stream=None):
    rows, cols = x.shape
    rc = lib().four_over_six_quantize(_ptr(x), _dtype(x), rows, cols, int(block), _ptr(S), int(objective), _ptr(w),
                                      int(w_row_stride), _ptr(codes), _ptr(sf_linear), _ptr(sf_swizzled),
                                      _ptr(block_loss), _stream(stream))
    _check("four_over_six_quantize", rc)


def nvfp4_dynamic_workspace() -> int:
    return int(lib().nvfp4_dynamic_workspace())


def scalesweep_quantize_dynamic(x, block: int, fp8_div: float, objective: int, w, w_row_stride: int, win_lo: int,
                                win_hi: int, S_out, status, workspace, codes, sf_linear=None, sf_swizzled=None,
                                block_loss=None, stream=None):
    rows, cols = x.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().scalesweep_quantize_dynamic(_ptr(x), _dtype(x), rows, cols, int(block), float(fp8_div), int(objective),
                                           _ptr(w), int(w_row_stride), int(win_lo), int(win_hi), _ptr(S_out),
                                           _ptr(status), _ptr(workspace), ws_bytes, _ptr(codes), _ptr(sf_linear),
                                           _ptr(sf_swizzled), _ptr(block_loss), _stream(stream))
    _check("scalesweep_quantize_dynamic", rc)


def absmax_quantize_dynamic(x, block: int, fp8_div: float, S_out, status, workspace, codes, sf_linear=None,
                            sf_swizzled=None, block_loss=None, stream=None):
    rows, cols = x.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().absmax_quantize_dynamic(_ptr(x), _dtype(x), rows, cols, int(block), float(fp8_div), _ptr(S_out),
                                       _ptr(status), _ptr(workspace), ws_bytes, _ptr(codes), _ptr(sf_linear),
                                       _ptr(sf_swizzled), _ptr(block_loss), _stream(stream))
    _check("absmax_quantize_dynamic", rc)


def scalesweep_quantize_group_workspace() -> int:
    return int(lib().scalesweep_quantize_group_workspace())


def group_descriptors(xs, ws, w_row_strides, codes, sf_linear, sf_swizzled):
    """The nvfp4_group_tensor array for tensors xs[i] with weights ws[i] (None
    for MSE) and output buffers codes[i], sf_linear[i], sf_swizzled[i] (None
    where not wanted).  Reusable across calls on the same buffers."""
    n = len(xs)
    arr = (GroupTensor * n)()
    for i, x in enumerate(xs):
        rows, cols = x.shape
        arr[i] = GroupTensor(x.data_ptr(), rows, cols, ws[i].data_ptr() if ws[i] is not None else None,
                             int(w_row_strides[i]), codes[i].data_ptr(),
                             sf_linear[i].data_ptr() if sf_linear[i] is not None else None,
                             sf_swizzled[i].data_ptr() if sf_swizzled[i] is not None else None)
    return arr


def scalesweep_quantize_group(desc, dtype: int, objective: int, fp8_div: float, S, status=None, workspace=None,
                              stream=None, block: int = 16, schedule: int | None = None):
    """desc: the array from group_descriptors.  fp8_div 0 reads S[i]; > 0
    computes and writes S[i] during the call.  schedule None calls
    scalesweep_quantize_group (the library's choice); an NVFP4_GROUP_SCHEDULE_*
    value calls scalesweep_quantize_group_scheduled with it."""
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    if schedule is None:
        rc = lib().scalesweep_quantize_group(desc, len(desc), int(dtype), int(block), int(objective), float(fp8_div),
                                             _ptr(S), _ptr(status), _ptr(workspace), ws_bytes, _stream(stream))
        _check("scalesweep_quantize_group", rc)
    else:
        rc = lib().scalesweep_quantize_group_scheduled(desc, len(desc), int(dtype), int(block), int(objective),
                                                       float(fp8_div), _ptr(S), _ptr(status), _ptr(workspace),
                                                       ws_bytes, int(schedule), _stream(stream))
        _check("scalesweep_quantize_group_scheduled", rc)


def absmax_quantize_group(desc, dtype: int, fp8_div: float, S, status=None, workspace=None, stream=None,
                          block: int = 16):
    """AbsMax over the tensors of desc in one launch (static or in-launch scales,
    as scalesweep_quantize_group)."""
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    rc = lib().absmax_quantize_group(desc, len(desc), int(dtype), int(block), float(fp8_div), _ptr(S),
                                     _ptr(status), _ptr(workspace), ws_bytes, _stream(stream))
    _check("absmax_quantize_group", rc)


def nvfp4_selftest_wait_timeout(which: int, x, S, status, workspace, codes, sf_linear, stream=None):
    """Makes the device waits of the dynamic-scale sweep (which = 0) or of the
    grouped launch (which = 1) run out; status bit 1 reports it."""
    rows, cols = x.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().nvfp4_selftest_wait_timeout(int(which), _ptr(x), rows, cols, _ptr(S), _ptr(status), _ptr(workspace),
                                           ws_bytes, _ptr(codes), _ptr(sf_linear), _stream(stream))
    _check("nvfp4_selftest_wait_timeout", rc)


def nvfp4_optimal_scale(x, block: int, S, objective: int, w, w_row_stride: int, s_opt, loss_opt, fp8_code=None,
                        loss_fp8=None, stream=None):
    rows, cols = x.shape
    rc = lib().nvfp4_optimal_scale(_ptr(x), _dtype(x), rows, cols, int(block), _ptr(S), int(objective), _ptr(w),
                                   int(w_row_stride), _ptr(s_opt), _ptr(loss_opt), _ptr(fp8_code), _ptr(loss_fp8),
                                   _stream(stream))
    _check("nvfp4_optimal_scale", rc)


def nvfp4_dequantize(codes, sf, layout: int, S, rows: int, cols: int, block: int, out, stream=None):
    rc = lib().nvfp4_dequantize(_ptr(codes), _ptr(sf), int(layout), _ptr(S), int(rows), int(cols), int(block),
                                _ptr(out), _dtype(out), _stream(stream))
    _check("nvfp4_dequantize", rc)


# --------------------------------------------------------------------------- buffer helpers
def swizzled_bytes(rows: int, cols: int, block: int = 16) -> int:
    kb = cols // block
    return -(-rows // 128) * 128 * (-(-kb // 4)) * 4


def empty_outputs(rows: int, cols: int, block: int, device="cuda", linear=True, swizzled=False, loss=False) -> dict:
    """Allocate the output buffers of a quantise call with torch (the library
    itself never allocates)."""
    out = {"codes": torch.empty(rows, cols // 2, dtype=torch.uint8, device=device)}
    out["sf_linear"] = torch.empty(rows, cols // block, dtype=torch.uint8, device=device) if linear else None
    out["sf_swizzled"] = torch.empty(swizzled_bytes(rows, cols, block), dtype=torch.uint8, device=device) \
        if swizzled else None
    out["block_loss"] = torch.empty(rows * (cols // block), dtype=torch.float32, device=device) if loss else None
    return out


def nvfp4_ldlq_prepare_workspace(n: int) -> int:
    return int(lib().nvfp4_ldlq_prepare_workspace(int(n)))


def nvfp4_ldlq_prepare(H, damp: float, perm, U, D, status=None, workspace=None, stream=None):
    """Damped, reordered UDU^T factor of the Hessian H [n, n] float32 for LDLQ:
    perm [n] int32, U [n, n] float32, D [n] float32 (outputs)."""
    n = H.shape[0]
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().nvfp4_ldlq_prepare(_ptr(H), n, float(damp), _ptr(perm), _ptr(U), _ptr(D), _ptr(status),
                                  _ptr(workspace), ws_bytes, _stream(stream))
    _check("nvfp4_ldlq_prepare", rc)


def nvfp4_ldlq_workspace(rows: int, cols: int) -> int:
    return int(lib().nvfp4_ldlq_workspace(int(rows), int(cols)))


def ldlq_quantize(W, block: int, S, sf_linear, perm, U, codes, status=None, workspace=None, stream=None):
    """LDLQ (GPTQ) quantization of W [rows, cols] with the fixed scales sf_linear,
    processing order perm and factor U from nvfp4_ldlq_prepare."""
    rows, cols = W.shape
    ws_bytes = workspace.numel() * workspace.element_size()
    rc = lib().ldlq_quantize(_ptr(W), _dtype(W), rows, cols, int(block), _ptr(S), _ptr(sf_linear), _ptr(perm),
                             _ptr(U), _ptr(codes), _ptr(status), _ptr(workspace), ws_bytes, _stream(stream))
    _check("ldlq_quantize", rc)


def nvfp4_row_shard_layout(rows: int, cols: int, block: int, world: int, rank: int) -> RowShard:
    """Rows and output offsets of shard `rank` of `world` (host-only, no GPU needed)."""
    out = RowShard()
    rc = lib().nvfp4_row_shard_layout(int(rows), int(cols), int(block), int(world), int(rank), ctypes.byref(out))
    _check("nvfp4_row_shard_layout", rc)
    return out
