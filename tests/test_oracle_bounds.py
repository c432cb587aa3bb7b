"""Pins of the oracle's bound machinery against what the paper prints.

The rational helpers in oracle/bounds.py must reproduce, exactly:
* the per-mantissa upper-bound table for alpha = 12/7 (Sec. 4.2.2 / Lemma 4.2),
* the per-mantissa lower-bound table for n = 16 (Sec. 4.2.2 / Lemma 4.3),
* the convex certificates A, B, A+15B of Appendix B.3,
* the legal ratios in (3/4, 4/5) of Appendix B.3,
* Lemma 4.2's +7 bound (and that it is attained).
A wrong grid point, midpoint, floor/ceil or exponent bias in the oracle shows
up as a wrong table entry here.
"""
import random
from fractions import Fraction as F

from conftest import golden_rows
from oracle import bounds


def _bits(s):
    return int(s, 2)


def test_upper_bound_table_closed_interval():
    want = [(_bits(b), _bits(sup), int(d)) for b, sup, d in golden_rows("upper_bound_table.txt")]
    assert bounds.upper_table(F(12, 7), closed=True) == want
    # the same table from other binades (the bound does not depend on the exponent field)
    for ef in (2, 5, 10):
        assert bounds.upper_table(F(12, 7), exponent_field=ef, closed=True) == want


def test_upper_bound_table_half_open_reading():
    """With s_base restricted to [v_b, v_{b+1}) the b = 101 entry drops to 6;
    the paper's 7 is the closed-interval (conservative) value."""
    want = [(_bits(b), _bits(sup), int(d)) for b, sup, d in golden_rows("upper_bound_table.txt")]
    got = bounds.upper_table(F(12, 7), closed=False)
    diff = [(w, g) for w, g in zip(want, got) if w != g]
    assert diff == [((5, 12, 7), (5, 11, 6))]


def test_lower_bound_table():
    want = [(_bits(b), _bits(inf), int(d)) for b, inf, d in golden_rows("lower_bound_table.txt")]
    assert bounds.lower_table(F(4, 5)) == want
    assert max(d for _, _, d in want) == 3   # the [-3, ...] MSE window


def test_convex_certificates():
    lam = [F(1, 4), F(1, 4), F(1, 2)]
    for row in (" ".join(r) for r in golden_rows("certificates.txt")):
        r_s, us_s, B_s, A_s, AB_s = [p.strip() for p in row.split("|")]
        r = F(r_s)
        us = [F(u) for u in us_s.split()]
        A, B = bounds.certificate(r, us, lam, m=r.denominator)
        assert B == F(B_s)
        assert A == F(A_s)
        assert A + 15 * B == F(AB_s)
        assert A + 15 * B <= 0
        assert all(u > r for u in us) and all(u <= F(11, 7) for u in us)


def test_r_le_three_quarters_excluded_by_doubling():
    """For r <= 3/4 the doubling argument: B_{2r,r} = r^2/4 and
    A_{2r,r} + 15 B_{2r,r} < 0 for every legal ratio (Appendix B.3)."""
    for r in sorted(x for x in bounds.normal_ratios() if F(1, 8) <= x <= F(3, 4)):
        A, B = bounds.certificate(r, [2 * r], [F(1)], m=8)
        assert B == r * r / 4
        assert A + 15 * B < 0


def test_legal_ratios():
    want = [F(x) for x in golden_rows("legal_ratios.txt")[0]]
    assert bounds.legal_ratios_in(F(3, 4), F(4, 5)) == sorted(want)


def test_lemma2_bound_and_tightness():
    rows = {r[0]: r[1] for r in golden_rows("windows.txt")}
    alpha = F(rows["lemma2_alpha"])
    assert bounds.lemma2_bound(alpha, 3) == int(rows["lemma2_bound"]) == 7
    assert bounds.lemma2_sup(alpha) == 7
    for a in (F(1), F(5, 4), F(3, 2), F(2)):
        assert bounds.lemma2_sup(a) <= bounds.lemma2_bound(a, 3)


def test_default_windows(oracle_mod):
    rows = {r[0]: (int(r[1]), int(r[2])) for r in golden_rows("windows.txt") if r[0] in ("mse", "wmse")}
    assert oracle_mod.default_window(oracle_mod.MSE, 16) == rows["mse"]
    assert oracle_mod.default_window(oracle_mod.WMSE, 16) == rows["wmse"]


def _loss_exact(s, xs, ws):
    tot = F(0)
    for x, w in zip(xs, ws):
        a = abs(x)
        best = min((a - s * g) ** 2 for g in bounds.GRID)
        tot += w * best
    return tot


def test_lemma1_scale_halving_exact():
    """Lemma 4.1: s > max|x| / 3.5  =>  L(s/2) <= L(s), checked exactly."""
    rnd = random.Random(7)
    for _ in range(400):
        n = rnd.choice([1, 4, 16])
        xs = [F(rnd.randint(-1000, 1000), 97) for _ in range(n)]
        ws = [F(rnd.randint(0, 50), 7) for _ in range(n)]
        m = max(abs(x) for x in xs)
        if m == 0:
            continue
        s = m / F(7, 2) * F(rnd.randint(1001, 3000), 1000)
        assert _loss_exact(s / 2, xs, ws) <= _loss_exact(s, xs, ws)
