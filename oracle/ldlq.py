"""LDLQ (GPTQ) with fixed NVFP4 block scales and static reordering -- oracle.

Test infrastructure only, like the rest of ``oracle/``: plain float64 numpy, no
code shared with the CUDA library.

What it computes (Appendix A.2, "GPTQ" paragraph, of the ScaleSweep paper):
GPTQ run as LDLQ (the QuIP form, algorithmically the same as GPTQ), damping of
0.01 x the mean of the Hessian diagonal, and MR-GPTQ's static reordering -- the
NVFP4 block scales are fixed before the error-feedback pass, and the input
channels are processed in descending order of the Hessian diagonal.

Notation.  W [m, n]: rows are output channels, columns input channels, NVFP4
blocks of 16 run along the columns.  H [n, n]: the input Gram matrix X^T X
(Sec. 3.3, the WMSE derivation; its diagonal is the importance Imp).  With pi
the processing order and H_pi the damped Hessian in that order,

    H_pi = (U + I) D (U + I)^T,   U strictly upper triangular, D diagonal > 0,

and LDLQ quantizes column k of W_pi after the columns before it:

    T_k  = W_k + sum_{i<k} (W_i - What_i) U_ik,      What_k = Q(T_k).

Q is NVFP4 rounding with the fixed block scale of the element's (original)
block, taken in the kernels' float32 contract: t = fl32(T), y = fl32(t*E) with
E = fl32(1/S), q = RNE_E2M1(fl32(y*fl32(1/v))) (saturating at 6, ties to the even
code), What = fl32(fl32(q*v)*S).  A block whose scale code is 0, or an unusable
global scale, quantizes to signed zeros (the sweep's zero rule).  A target that
is exactly zero takes the +0 code: the sign of a zero sum depends on the
summation order, which neither side fixes (reading; LDLQ itself is silent).

The same result in GPTQ's own form (error feedback through the upper Cholesky
factor of the inverse Hessian) is ``gptq``; the two are independent
formulations and pin each other.
"""
from __future__ import annotations

import numpy as np

E2M1_GRID = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])


def e4m3_value(code):
    """Exact value of E4M3 codes (bias 7; codes 1..7 are subnormal, c * 2^-9)."""
    c = np.asarray(code, dtype=np.int64)
    e, m = c >> 3, c & 7
    normal = np.ldexp(1.0 + m / 8.0, (e - 7).astype(np.int64))
    sub = c * 2.0 ** -9
    return np.where(e > 0, normal, sub)


def rne_e2m1(a):
    """Code 0..7 of the E2M1 magnitude nearest to a >= 0 (float32 values);
    ties go to the even code, anything at or above 6 saturates to 6."""
    a = np.asarray(a, dtype=np.float64)
    d = np.abs(a[..., None] - E2M1_GRID)
    dmin = d.min(axis=-1, keepdims=True)
    tied = d == dmin
    even = tied & (np.arange(8) % 2 == 0)
    k = np.where(even.any(axis=-1), np.argmax(even, axis=-1), np.argmax(tied, axis=-1))
    return np.where(a >= 6.0, 7, k).astype(np.int64)


def quantize_fixed(t, S, code, zero_positive=False):
    """Q(t) with fixed E4M3 scale codes: returns (nibbles, dequantized values).

    t: float64 targets; code: per-element scale codes (0..126); zero_positive:
    an exactly zero y takes the +0 code (LDLQ targets), else its own sign (the
    sweep's rounding of inputs)."""
    t32 = np.asarray(t, dtype=np.float64).astype(np.float32)
    S32 = np.float32(S)
    with np.errstate(divide="ignore", over="ignore", invalid="ignore"):
        E = np.float32(1.0) / S32
    usable = bool(S32 > 0 and np.isfinite(S32) and np.isfinite(E))
    code = np.asarray(code, dtype=np.int64)
    y = (t32 * E).astype(np.float32) if usable else t32
    sign = np.signbit(y)
    if zero_positive:
        sign = sign & (y != 0)
    zero = (code == 0) | (not usable)
    v = e4m3_value(np.where(zero, 1, code)).astype(np.float32)
    r = (np.float32(1.0) / v).astype(np.float32)
    with np.errstate(over="ignore", invalid="ignore"):
        tq = (y * r).astype(np.float32)
    k = np.where(zero, 0, rne_e2m1(np.abs(tq)))
    nib = (sign.astype(np.int64) << 3) | k
    q = E2M1_GRID[k] * np.where(sign, -1.0, 1.0)
    qv = (q.astype(np.float32) * v).astype(np.float32)          # exact (<= 6 significant bits)
    val = (qv * S32).astype(np.float32) if usable else np.zeros_like(qv)
    val = np.where(zero, np.where(sign, -0.0, 0.0), val.astype(np.float64))
    return nib, val


def damp_and_order(H, alpha=0.01):
    """Damped Hessian H + alpha*mean(diag H)*I and the static processing order:
    input channels by descending Hessian diagonal, ties by ascending index."""
    H = np.asarray(H, dtype=np.float64)
    n = H.shape[0]
    lam = alpha * float(np.mean(np.diag(H)))
    Hd = H + lam * np.eye(n)
    perm = np.array(sorted(range(n), key=lambda i: (-H[i, i], i)), dtype=np.int64)
    return Hd, perm


def udu(Hp):
    """Hp = (U + I) D (U + I)^T with U strictly upper triangular: the Cholesky
    factor of the index-reversed matrix, reversed back (J L J is upper)."""
    n = Hp.shape[0]
    J = np.arange(n)[::-1]
    L = np.linalg.cholesky(Hp[np.ix_(J, J)])
    Rt = L[np.ix_(J, J)]                                         # upper, Hp = Rt Rt^T
    d = np.diag(Rt)
    U = Rt / d[None, :] - np.eye(n)
    return np.triu(U, 1), d * d


def ldlq(W, H, S, sf, block=16, alpha=0.01):
    """LDLQ with fixed scale codes sf [m, n/block] (original column order).

    Returns a dict: nib [m, n] nibbles and What [m, n] values in the original
    column order, perm, U, D (processing order) and T [m, n] the targets in
    processing order."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    Hd, perm = damp_and_order(H, alpha)
    U, D = udu(Hd[np.ix_(perm, perm)])
    Wp = W[:, perm]
    code_el = np.asarray(sf, dtype=np.int64)[:, perm // block]
    What = np.zeros((m, n))
    nib = np.zeros((m, n), dtype=np.int64)
    T = np.zeros((m, n))
    for k in range(n):
        T[:, k] = Wp[:, k] + (Wp[:, :k] - What[:, :k]) @ U[:k, k]
        nib[:, k], What[:, k] = quantize_fixed(T[:, k], S, code_el[:, k], zero_positive=True)
    inv = np.empty(n, dtype=np.int64)
    inv[perm] = np.arange(n)
    return {"nib": nib[:, inv], "What": What[:, inv], "perm": perm, "U": U, "D": D, "T": T}


def gptq(W, H, S, sf, block=16, alpha=0.01):
    """The same quantization in GPTQ's form: columns in processing order,
    err_i = (w_i - What_i) / R_ii and w_j -= err_i R_ij for j > i, with R the
    upper Cholesky factor of the inverse damped Hessian (H^-1 = R^T R)."""
    W = np.asarray(W, dtype=np.float64)
    m, n = W.shape
    Hd, perm = damp_and_order(H, alpha)
    R = np.linalg.cholesky(np.linalg.inv(Hd[np.ix_(perm, perm)])).T
    Wt = W[:, perm].copy()
    code_el = np.asarray(sf, dtype=np.int64)[:, perm // block]
    What = np.zeros((m, n))
    nib = np.zeros((m, n), dtype=np.int64)
    for i in range(n):
        nib[:, i], What[:, i] = quantize_fixed(Wt[:, i], S, code_el[:, i], zero_positive=True)
        err = (Wt[:, i] - What[:, i]) / R[i, i]
        Wt[:, i + 1:] -= np.outer(err, R[i, i + 1:])
    inv = np.empty(n, dtype=np.int64)
    inv[perm] = np.arange(n)
    return {"nib": nib[:, inv], "What": What[:, inv], "perm": perm}


def targets(W, What, perm, U):
    """LDLQ targets in processing order for given reconstructions What (original
    order): T = W_pi + (W_pi - What_pi) U.  Row r of T depends only on row r."""
    W = np.asarray(W, dtype=np.float64)
    Wp, Hp_ = W[:, perm], np.asarray(What, dtype=np.float64)[:, perm]
    return Wp + (Wp - Hp_) @ U


def proxy_loss(W, What, H):
    """tr((W - What) H (W - What)^T): the layer-output error X (W - What)^T
    summed over calibration rows (Sec. 3.3)."""
    E = np.asarray(W, dtype=np.float64) - np.asarray(What, dtype=np.float64)
    return float(np.einsum("ij,jk,ik->", E, np.asarray(H, dtype=np.float64), E))


def decision_margin(T, S, code):
    """Distance of |fl32(fl32(T)*E) * fl32(1/v)| from the nearest E2M1 rounding
    boundary (midpoint), relative to max(1, value): small margins are where a
    float32 and a float64 accumulation of T may round differently."""
    t32 = np.asarray(T, dtype=np.float64).astype(np.float32)
    with np.errstate(divide="ignore", over="ignore", invalid="ignore"):
        E = np.float32(1.0) / np.float32(S)
        v = e4m3_value(np.where(np.asarray(code) == 0, 1, code)).astype(np.float32)
        z = np.abs(((t32 * E).astype(np.float32) * (np.float32(1.0) / v)).astype(np.float32)).astype(np.float64)
        mids = np.array([0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0])
        return np.min(np.abs(z[..., None] - mids), axis=-1) / np.maximum(1.0, z)
