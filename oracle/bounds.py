"""Exact rational re-derivation of ScaleSweep's sweep bounds -- test infrastructure.

Everything is computed with ``fractions.Fraction`` straight from the format
definitions, so the tables the paper prints can be checked against it:

* E4M3 values from the EeMm formula of Appendix A (bias 7, subnormals for a=0),
  codes 1..126 positive finite (0x7F is NaN);
* the per-mantissa upper bound for alpha = 12/7 (Lemma 4.2 and the upper-bound
  table of Sec. 4.2.2) and the per-mantissa lower bound ceil_FP8((4/5) s0)
  (Lemma 4.3 and the lower-bound table of Sec. 4.2.2);
* the single-coordinate loss d_r(y) = min_g (y - r g)^2 over the non-negative
  E2M1 grid and the convex certificates A, B, A+15B of the proof of Lemma 4.3
  (Appendix B.3), evaluated exactly at the breakpoints of the piecewise-affine
  difference;
* the enumeration of legal E4M3 ratios in (3/4, 4/5) (Appendix B.3).
"""
from __future__ import annotations

from fractions import Fraction as F
from math import ceil

# Non-negative E2M1 grid (Sec. 3.2); midpoints between consecutive points.
GRID = [F(0), F(1, 2), F(1), F(3, 2), F(2), F(3), F(4), F(6)]
MIDPOINTS = [(GRID[k] + GRID[k + 1]) / 2 for k in range(7)]


def eemm_value(e: int, m: int, code: int) -> F:
    """Appendix A: v(c,a,b) for an EeMm code, bias 2^(e-1)-1."""
    M = 1 << m
    c = (code >> (e + m)) & 1
    a = (code >> m) & ((1 << e) - 1)
    b = code & (M - 1)
    bias = (1 << (e - 1)) - 1
    if a != 0:
        v = F(2) ** (a - bias) * (1 + F(b, M))
    else:
        v = F(2) ** (1 - bias) * F(b, M)
    return -v if c else v


E4M3 = [(c, eemm_value(4, 3, c)) for c in range(0, 127)]   # code 127 is NaN
E4M3_POS = E4M3[1:]
E2M1 = [eemm_value(2, 1, c) for c in range(16)]


def floor_fp8(x: F) -> tuple[int, F]:
    """Largest E4M3 (code, value) with value <= x (code 0 if none is positive)."""
    best = E4M3[0]
    for c, v in E4M3:
        if v <= x:
            best = (c, v)
    return best


def ceil_fp8(x: F) -> tuple[int, F]:
    """Smallest positive E4M3 (code, value) with value >= x (None past 448)."""
    for c, v in E4M3_POS:
        if v >= x:
            return (c, v)
    return None


def pred_fp8(x: F) -> tuple[int, F]:
    """Largest E4M3 value strictly below x."""
    best = E4M3[0]
    for c, v in E4M3:
        if v < x:
            best = (c, v)
    return best


def lemma2_bound(alpha: F, m: int) -> int:
    """Lemma 4.2 right-hand side ceil((1 - 1/alpha) 2^(m+1))."""
    return ceil((1 - 1 / alpha) * 2 ** (m + 1))


def lemma2_sup(alpha: F) -> int:
    """max over positive x of I(floor(alpha x)) - I(floor(x)) in E4M3, by
    evaluating at every jump point of the two step functions (both are
    right-continuous and piecewise constant)."""
    pts = set()
    for _, v in E4M3_POS:
        pts.add(v)
        pts.add(v / alpha)
    best = -10 ** 9
    for x in pts:
        if x <= 0:
            continue
        c1, _ = floor_fp8(x)
        if c1 == 0:
            continue
        c2, v2 = floor_fp8(alpha * x)
        if alpha * x > E4M3_POS[-1][1]:
            continue  # past the top of the format: the lemma is about finite values
        best = max(best, c2 - c1)
    return best


def upper_table(alpha: F = F(12, 7), exponent_field: int = 7, closed: bool = True) -> list[tuple[int, int, int]]:
    """Per-mantissa upper bound: for s_base^FP8 with mantissa b, the carry bit
    and mantissa of the largest floor_FP8(alpha * s_base) over
    s_base in [v_b, v_{b+1}] (closed) or [v_b, v_{b+1}) (half-open).
    Returns (b, sup, delta) with sup = code(floor) - 8*exponent_field."""
    out = []
    for b in range(8):
        code = exponent_field * 8 + b
        v_next = eemm_value(4, 3, code + 1)
        if closed:
            c_top, _ = floor_fp8(alpha * v_next)
        else:
            c_top, _ = pred_fp8(alpha * v_next)
            c_at, _ = floor_fp8(alpha * v_next)
            if alpha * v_next != eemm_value(4, 3, c_at):
                c_top = c_at
        sup = c_top - exponent_field * 8
        out.append((b, sup, sup - b))
    return out


def lower_table(ratio: F = F(4, 5), exponent_field: int = 7) -> list[tuple[int, int, int]]:
    """Per-mantissa lower bound: borrow bit and mantissa of ceil_FP8(ratio * s0)
    for s0 with mantissa b.  Returns (b, inf, delta) with inf = code(ceil) -
    8*(exponent_field-1) - 8 encoded as borrow*8 + mantissa, and delta = b - rel
    where rel = code(ceil) - 8*exponent_field."""
    out = []
    for b in range(8):
        s0 = eemm_value(4, 3, exponent_field * 8 + b)
        c, _ = ceil_fp8(ratio * s0)
        rel = c - exponent_field * 8            # negative when it borrows
        inf = rel + 16 if rel < 0 else rel      # borrow bit then 3 mantissa bits
        out.append((b, inf, b - rel))
    return out


def d_r(r: F, y: F) -> F:
    """Single-coordinate loss min_g (y - r g)^2 over the non-negative grid."""
    return min((y - r * g) ** 2 for g in GRID)


def certificate(r: F, us: list[F], lams: list[F], m: int) -> tuple[F, F]:
    """A = sup_{6<=y<=6rho} Delta(y), B = sup_{0<=y<=6rho} Delta(y) with
    Delta = sum_j lam_j d_{u_j} - d_r and rho = (m+1)/m.  Delta is piecewise
    affine (the y^2 terms cancel) so the sups are attained at breakpoints."""
    rho = F(m + 1, m)
    top = 6 * rho
    bps = {F(0), F(6), top}
    for s in [r] + list(us):
        for mu in MIDPOINTS:
            bps.add(s * mu)

    def delta(y: F) -> F:
        return sum(l * d_r(u, y) for u, l in zip(us, lams)) - d_r(r, y)

    B = max(delta(y) for y in bps if 0 <= y <= top)
    A = max(delta(y) for y in bps if 6 <= y <= top)
    return A, B


def normal_ratios() -> set[F]:
    """All ratios v/v' of positive normal E4M3 values (significands m/8, m in 8..15)."""
    out = set()
    for j in range(8, 16):
        for mm in range(8, 16):
            for da in range(-3, 4):
                out.add(F(j, mm) * F(2) ** da)
    return out


def legal_ratios_in(lo: F, hi: F) -> list[F]:
    return sorted(r for r in normal_ratios() if lo < r < hi)
