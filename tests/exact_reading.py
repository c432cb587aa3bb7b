"""ScaleSweep under exact rounding of x/S and x/(S v_c): the paper's own
statement of the sweep (Sec. 3.2 rounds x/S and x/s exactly; Sec. 4.2.2
sweeps the window around floor_E4M3(max|x| / (6 S))), without the float32
arithmetic contract the kernels and the oracle share.

Every decision is taken exactly in float64: the floor code I0 compares
6 S v_c (at most 30 significant bits) with max|x|, and each E2M1 rounding
compares |x| with mu S v_c for the grid midpoints mu (at most 31 bits), so
no rounding enters; ties of the E2M1 rounding go to the even code.  Losses
sum w (x - q v S)^2, which is S^2 times the S-normalised loss, in float64.

Used by test_oracle_contract_reading.py to count how many blocks the float32
contract quantises differently from this exact reading.  Test code only: it
holds no CUDA path and is not imported by the oracle.
"""
from __future__ import annotations

import numpy as np

from oracle import bounds

MIDS = (0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0)
MIDS_ARR = np.array(MIDS)
GRID = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])
V = np.array([float(v) for _, v in bounds.E4M3], dtype=np.float64)      # codes 0..126, exact values


def quantize_exact(x: np.ndarray, S: float, block: int, window: tuple[int, int], w: np.ndarray | None = None,
                   chunk_blocks: int = 1 << 18):
    """Codes [rows, cols/2] and scale codes [rows, cols/block] of the exact
    reading; w is a per-column weight vector (WMSE) or None (MSE)."""
    rows, cols = x.shape
    kb = cols // block
    X = np.ascontiguousarray(x, dtype=np.float32).astype(np.float64).reshape(-1, block)
    nb = X.shape[0]
    Wb = None if w is None else np.tile(np.asarray(w, np.float64).reshape(kb, block), (rows, 1))
    S64 = float(np.float32(S))
    thr = 6.0 * S64 * V                                        # exact: 6 S v_c
    sf = np.zeros(nb, np.uint8)
    nib = np.zeros((nb, block), np.uint8)
    lo, hi = window
    for b0 in range(0, nb, chunk_blocks):
        Xc = X[b0:b0 + chunk_blocks]
        Wc = None if Wb is None else Wb[b0:b0 + chunk_blocks]
        A = np.abs(Xc)
        sign = np.signbit(Xc).astype(np.uint8) << 3
        amax = A.max(axis=1)
        I0 = np.searchsorted(thr, amax, side="right") - 1       # largest c with 6 S v_c <= max|x|
        I0 = np.minimum(I0, 126)
        clo = np.clip(I0 + lo, 1, 126)
        chi = np.clip(I0 + hi, 1, 126)
        best = np.full(Xc.shape[0], np.inf)
        bestc = clo.copy()
        bestq = np.zeros(Xc.shape, np.uint8)
        for k in range(hi - lo + 1):
            c = clo + k
            live = c <= chi
            vS = (V[np.minimum(c, 126)] * S64)[:, None]         # exact: v_c S
            # |x| / (v S) rounded to float64 is monotone in |x|, so it decides
            # every midpoint exactly except where it lands on one; there the
            # exact comparison with mu v S (a tie rounds to the even code) does
            q = A / vS
            idx = np.searchsorted(MIDS_ARR, q, side="left").astype(np.uint8)
            on = np.nonzero(MIDS_ARR[np.minimum(idx, 6)] == q)    # q is exactly midpoint j = idx
            if on[0].size:
                j = idx[on]
                t = MIDS_ARR[j] * vS[on[0], 0]
                a = A[on]
                idx[on] += (a > t) | ((a == t) & (j % 2 == 1))
            e = Xc - np.copysign(GRID[idx], Xc) * vS
            L = (e * e if Wc is None else Wc * e * e).sum(axis=1)
            better = live & (L < best)
            best = np.where(better, L, best)
            bestc = np.where(better, c, bestc)
            bestq = np.where(better[:, None], idx, bestq)
        zero = amax == 0
        bestc = np.where(zero, 0, bestc)
        bestq = np.where(zero[:, None], 0, bestq)
        sf[b0:b0 + Xc.shape[0]] = bestc
        nib[b0:b0 + Xc.shape[0]] = bestq | sign
    codes = (nib[:, 0::2] | (nib[:, 1::2] << 4)).reshape(rows, cols // 2)
    return codes, sf.reshape(rows, kb)
