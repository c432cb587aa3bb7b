"""CPU oracle for NVFP4 ScaleSweep quantisation -- test infrastructure only.

Only ``tests/``, ``__graft_entry__.smoke()`` and the cpu_baseline / reference
legs of ``bench.py`` may import this package.  It shares no code with the CUDA
library in ``paper_2606_07618_gb300`` and never imports it.

The arithmetic lives in ``nvfp4_oracle.c`` (plain scalar C, float64 losses,
float32 for the rounding decisions the kernels also take in float32); this
module builds it with gcc and wraps it for numpy arrays.  ``bounds.py`` holds
the exact rational re-derivations of the paper's bit-pattern bounds.

``swizzle_scales`` (the 128x4 scale-factor layout, defined by NVIDIA's block-scaling
layout rather than by the paper) is pinned on the GPU against cuBLASLt's NVFP4
block-scaled GEMM.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import sys

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "nvfp4_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

METHOD_SCALESWEEP, METHOD_ABSMAX, METHOD_FOUR_SIX = 0, 1, 2
MSE, WMSE = 0, 1
LAYOUT_LINEAR, LAYOUT_SWIZZLED = 1, 2


def build(force: bool = False, openmp: bool = True) -> str:
    """Compile the oracle into oracle/liboracle.so (gcc, no FMA contraction)."""
    if not force and os.path.exists(_LIB_PATH) and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-fno-fast-math"]
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmds = ([base + ["-fopenmp", _SRC, "-o", tmp, "-lm"]] if openmp else []) + [base + [_SRC, "-o", tmp, "-lm"]]
    err = None
    for cmd in cmds:
        r = subprocess.run(cmd, capture_output=True, text=True)
        if r.returncode == 0:
            os.replace(tmp, _LIB_PATH)
            return _LIB_PATH
        err = r.stderr
    raise RuntimeError(f"oracle build failed: {err}")


def _load(path: str) -> ctypes.CDLL:
    L = ctypes.CDLL(path)
    c_i, c_i64, c_f, c_d, c_p = ctypes.c_int, ctypes.c_int64, ctypes.c_float, ctypes.c_double, ctypes.c_void_p
    L.oracle_e2m1_value.argtypes, L.oracle_e2m1_value.restype = [c_i], c_d
    L.oracle_e4m3_value.argtypes, L.oracle_e4m3_value.restype = [c_i], c_d
    L.oracle_e2m1_rne.argtypes, L.oracle_e2m1_rne.restype = [c_f], c_i
    L.oracle_e4m3_floor.argtypes, L.oracle_e4m3_floor.restype = [c_f], c_i
    L.oracle_e4m3_rn.argtypes, L.oracle_e4m3_rn.restype = [c_f], c_i
    L.oracle_global_scale.argtypes = [c_p, c_i64, c_f, c_p, c_p]
    L.oracle_quantize.argtypes = [c_i, c_p, c_i64, c_i64, c_i, c_f, c_i, c_p, c_i64, c_i, c_i,
                                  c_p, c_p, c_p, c_p, c_p, c_i, c_p, c_i]
    L.oracle_block_losses_at.argtypes = [c_p, c_i64, c_i64, c_i, c_f, c_i, c_p, c_i64, c_p, c_p, c_p, c_i]
    L.oracle_swizzle_offset.argtypes, L.oracle_swizzle_offset.restype = [c_i64, c_i64, c_i64], c_i64
    L.oracle_swizzle_bytes.argtypes, L.oracle_swizzle_bytes.restype = [c_i64, c_i64], c_i64
    L.oracle_swizzle_scales.argtypes = [c_p, c_i64, c_i64, c_p]
    L.oracle_dequantize.argtypes = [c_p, c_p, c_i, c_f, c_i64, c_i64, c_i, c_p, c_p]
    L.oracle_opt_scale.argtypes = [c_p, c_p, c_i, c_p, c_p]
    L.oracle_fp8_opt_code.argtypes = [c_p, c_p, c_i, c_d, c_p, c_p]
    return L


def lib() -> ctypes.CDLL:
    global _lib
    if _lib is None:
        build()
        _lib = _load(_LIB_PATH)
    return _lib


def build_variant(src_text: str, out_path: str) -> str:
    """Compile an edited copy of the oracle source (used by the planted-mistake
    tests to show that the pins catch plausible errors)."""
    src = out_path + ".c"
    with open(src, "w") as f:
        f.write(src_text)
    cmd = ["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", src, "-o", out_path, "-lm"]
    r = subprocess.run(cmd, capture_output=True, text=True)
    if r.returncode != 0:
        raise RuntimeError(r.stderr)
    return out_path


def swap_library(path: str | None):
    """Point this module at another build of the oracle (None restores the
    default); returns the previous handle."""
    global _lib
    prev = _lib
    _lib = _load(path) if path else None
    return prev


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


# --------------------------------------------------------------------------- formats
def e2m1_value(code: int) -> float:
    return lib().oracle_e2m1_value(int(code))


def e4m3_value(code: int) -> float:
    return lib().oracle_e4m3_value(int(code))


def e2m1_rne(t: float) -> int:
    return lib().oracle_e2m1_rne(float(t))


def e4m3_floor(s: float) -> int:
    return lib().oracle_e4m3_floor(float(s))


def e4m3_rn(s: float) -> int:
    return lib().oracle_e4m3_rn(float(s))


def default_window(objective: int, block: int) -> tuple[int, int]:
    """Bit-pattern offsets around I0 (Sec. 4.2.2): MSE [-3, 7] for 16-element
    blocks (Lemma 4.3 is proven for n = 16), WMSE [-8, 7].  Blocks of 32/64 use
    [-8, 7] for both objectives (the paper gives no window for them)."""
    if objective == MSE and block == 16:
        return (-3, 7)
    return (-8, 7)


# --------------------------------------------------------------------------- tensor ops
def global_scale(x: np.ndarray, D: float) -> tuple[float, bool]:
    """S = fl32(amax / fl32(6*D)); also reports whether x holds NaN/inf."""
    x = np.ascontiguousarray(x, dtype=np.float32).reshape(-1)
    S = np.zeros(1, np.float32)
    bad = np.zeros(1, np.int32)
    lib().oracle_global_scale(_ptr(x), x.size, float(D), _ptr(S), _ptr(bad))
    return float(S[0]), bool(bad[0])


def quantize(method: int, x: np.ndarray, block: int, S: float, objective: int = MSE,
             w: np.ndarray | None = None, w_row_stride: int = 0, window: tuple[int, int] | None = None,
             want_cand: bool = False, cand_stride: int = 16, nthreads: int = 0) -> dict:
    """Quantise a 2-D float32 array.  Returns codes [rows, cols/2] u8, sf
    [rows, cols/block] u8, best/second float64 per block and optionally the
    per-candidate losses."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    rows, cols = x.shape
    kb = cols // block
    if window is None:
        window = default_window(objective, block)
    codes = np.zeros((rows, cols // 2), np.uint8)
    sf = np.zeros((rows, kb), np.uint8)
    best = np.zeros(rows * kb, np.float64)
    second = np.zeros(rows * kb, np.float64)
    cand = np.zeros((rows * kb, cand_stride), np.float64) if want_cand else None
    cand_lo = np.zeros(rows * kb, np.int32) if want_cand else None
    if w is not None:
        w = np.ascontiguousarray(w, dtype=np.float32)
    rc = lib().oracle_quantize(method, _ptr(x), rows, cols, block, float(np.float32(S)), objective,
                               _ptr(w), int(w_row_stride), int(window[0]), int(window[1]),
                               _ptr(codes), _ptr(sf), _ptr(best), _ptr(second), _ptr(cand),
                               cand_stride, _ptr(cand_lo), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_quantize: bad arguments")
    out = dict(codes=codes, sf=sf, best=best, second=second)
    if want_cand:
        out["cand"], out["cand_lo"] = cand, cand_lo
    return out


def block_losses_at(x: np.ndarray, block: int, S: float, sf_codes: np.ndarray, objective: int = MSE,
                    w: np.ndarray | None = None, w_row_stride: int = 0, nthreads: int = 0,
                    want_codes: bool = False):
    """float64 loss of each block under the given scale codes (same contract);
    with want_codes also the packed nibbles those scales produce."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    rows, cols = x.shape
    sfc = np.ascontiguousarray(sf_codes, dtype=np.uint8).reshape(-1)
    out = np.zeros(rows * (cols // block), np.float64)
    codes = np.zeros((rows, cols // 2), np.uint8) if want_codes else None
    if w is not None:
        w = np.ascontiguousarray(w, dtype=np.float32)
    rc = lib().oracle_block_losses_at(_ptr(x), rows, cols, block, float(np.float32(S)), objective, _ptr(w),
                                      int(w_row_stride), _ptr(sfc), _ptr(out), _ptr(codes), int(nthreads))
    if rc != 0:
        raise ValueError("oracle_block_losses_at: bad arguments")
    return (out, codes) if want_codes else out


def swizzle_bytes(rows: int, kblocks: int) -> int:
    return lib().oracle_swizzle_bytes(rows, kblocks)


def swizzle_offset(r: int, k: int, kblocks: int) -> int:
    return lib().oracle_swizzle_offset(r, k, kblocks)


def swizzle_scales(sf_linear: np.ndarray) -> np.ndarray:
    sf_linear = np.ascontiguousarray(sf_linear, dtype=np.uint8)
    rows, kb = sf_linear.shape
    out = np.zeros(swizzle_bytes(rows, kb), np.uint8)
    lib().oracle_swizzle_scales(_ptr(sf_linear), rows, kb, _ptr(out))
    return out


def dequantize(codes: np.ndarray, sf: np.ndarray, layout: int, S: float, rows: int, cols: int, block: int,
               out_bf16: bool = False) -> np.ndarray:
    """x_hat = fl32(fl32(q*v)*S); bf16 output is the RNE of that fp32 value
    (returned as uint16 bit patterns)."""
    codes = np.ascontiguousarray(codes, dtype=np.uint8)
    sf = np.ascontiguousarray(sf, dtype=np.uint8)
    if out_bf16:
        out = np.zeros((rows, cols), np.uint16)
        rc = lib().oracle_dequantize(_ptr(codes), _ptr(sf), layout, float(np.float32(S)), rows, cols, block,
                                     None, _ptr(out))
    else:
        out = np.zeros((rows, cols), np.float32)
        rc = lib().oracle_dequantize(_ptr(codes), _ptr(sf), layout, float(np.float32(S)), rows, cols, block,
                                     _ptr(out), None)
    if rc != 0:
        raise ValueError("oracle_dequantize: bad arguments")
    return out


def opt_scale(y: np.ndarray, w: np.ndarray | None = None) -> tuple[float, float]:
    """Appendix C optimum (s*, L(s*)) of one block in the S-normalised domain."""
    y = np.ascontiguousarray(y, dtype=np.float32).reshape(-1)
    if w is not None:
        w = np.ascontiguousarray(w, dtype=np.float32).reshape(-1)
    s = np.zeros(1, np.float64)
    L = np.zeros(1, np.float64)
    lib().oracle_opt_scale(_ptr(y), _ptr(w), y.size, _ptr(s), _ptr(L))
    return float(s[0]), float(L[0])


def fp8_opt_code(y: np.ndarray, w: np.ndarray | None, s_opt: float) -> tuple[int, float]:
    y = np.ascontiguousarray(y, dtype=np.float32).reshape(-1)
    if w is not None:
        w = np.ascontiguousarray(w, dtype=np.float32).reshape(-1)
    c = np.zeros(1, np.int32)
    L = np.zeros(1, np.float64)
    lib().oracle_fp8_opt_code(_ptr(y), _ptr(w), y.size, float(s_opt), _ptr(c), _ptr(L))
    return int(c[0]), float(L[0])


def bf16_bits_to_f32(u16: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float32."""
    return (np.asarray(u16, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


if __name__ == "__main__":  # pragma: no cover
    print(build(force="--force" in sys.argv))
