"""Pins of the oracle's number formats against the paper and library routines.

* E2M1 grid: the set printed in Sec. 3.2 (golden/e2m1_grid.txt).
* E4M3: 126 positive finite values, max 448, bias 7 (Sec. 3.2, Sec. 4.2.2,
  Appendix A; golden/e4m3_facts.txt), cross-checked against torch's
  float8_e4m3fn decoding and against the rational Appendix-A formula.
* Rounding: RNE to E2M1 by brute force over the grid; floor/RN to E4M3 against
  the rational table and against torch's float8_e4m3fn (RNE) conversion.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch

from conftest import golden_rows
from oracle import bounds


def test_e2m1_grid_is_the_printed_set(oracle_mod):
    grid = [float(v) for v in golden_rows("e2m1_grid.txt")[0]]
    vals = [oracle_mod.e2m1_value(c) for c in range(8)]
    assert vals == grid
    neg = [oracle_mod.e2m1_value(8 + c) for c in range(8)]
    assert neg == [-g for g in grid]
    assert math.copysign(1.0, oracle_mod.e2m1_value(8)) == -1.0
    assert max(vals) == 6.0


def test_e4m3_facts(oracle_mod):
    facts = {r[0]: float(r[1]) for r in golden_rows("e4m3_facts.txt")}
    vals = [oracle_mod.e4m3_value(c) for c in range(127)]
    pos = [v for v in vals if v > 0]
    assert len(pos) == int(facts["positive_finite_count"])
    assert max(pos) == facts["max"] == vals[126]
    assert min(pos) == facts["min_subnormal"] == vals[1]
    assert vals[8] == facts["min_normal"]
    assert all(a < b for a, b in zip(vals, vals[1:])), "codes must order like values"
    assert math.isnan(oracle_mod.e4m3_value(127))
    assert math.isnan(oracle_mod.e4m3_value(255))


def test_e4m3_against_rational_formula(oracle_mod):
    for c, v in bounds.E4M3:
        assert oracle_mod.e4m3_value(c) == float(v)
        assert oracle_mod.e4m3_value(c | 0x80) == -float(v)
    for c in range(16):
        assert oracle_mod.e2m1_value(c) == float(bounds.E2M1[c])


def test_e4m3_against_torch_float8(oracle_mod):
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    tv = codes.view(torch.float8_e4m3fn).to(torch.float32).numpy()
    for c in range(256):
        ov = oracle_mod.e4m3_value(c)
        if math.isnan(ov):
            assert math.isnan(tv[c])
        else:
            assert ov == float(tv[c]), c


def _rne_bruteforce(t: float) -> int:
    grid = [Fraction(g) for g in (0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0)]
    a = abs(Fraction(t))
    d = [abs(a - g) for g in grid]
    m = min(d)
    ks = [k for k in range(8) if d[k] == m]
    k = ks[0] if len(ks) == 1 else [k for k in ks if k % 2 == 0][0]
    return (8 if math.copysign(1.0, t) < 0 else 0) | k


def test_e2m1_rne_bruteforce(oracle_mod):
    rng = np.random.default_rng(1)
    ts = list(rng.uniform(-8, 8, 20000).astype(np.float32))
    ts += list(rng.standard_normal(2000).astype(np.float32) * 1e-3)
    mids = [0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 7.0]
    for mu in mids:
        for v in (mu, np.nextafter(np.float32(mu), np.float32(0)), np.nextafter(np.float32(mu), np.float32(9))):
            ts += [np.float32(v), -np.float32(v)]
    ts += [np.float32(0.0), np.float32(-0.0), np.float32(6.0), np.float32(1e30), np.float32(-1e30)]
    for t in ts:
        assert oracle_mod.e2m1_rne(float(t)) == _rne_bruteforce(float(t)), t
    # ties go to the even code: 0.25->0, 0.75->1, 1.25->1, 1.75->2, 2.5->2, 3.5->4, 5->4
    expect = {0.25: 0.0, 0.75: 1.0, 1.25: 1.0, 1.75: 2.0, 2.5: 2.0, 3.5: 4.0, 5.0: 4.0}
    for t, q in expect.items():
        assert oracle_mod.e2m1_value(oracle_mod.e2m1_rne(t)) == q
    assert oracle_mod.e2m1_rne(-0.1) == 8  # negative values rounding to zero keep the sign


def test_e4m3_floor_against_rational(oracle_mod):
    rng = np.random.default_rng(2)
    ss = list(np.exp(rng.uniform(math.log(1e-4), math.log(600), 4000)).astype(np.float32))
    ss += [np.float32(v) for _, v in bounds.E4M3_POS]
    ss += [np.nextafter(np.float32(v), np.float32(0)) for _, v in bounds.E4M3_POS]
    ss += [np.float32(0.0), np.float32(1e-12), np.float32(448.0), np.float32(1e6)]
    for s in ss:
        c, _ = bounds.floor_fp8(Fraction(float(s)))
        assert oracle_mod.e4m3_floor(float(s)) == c, s


def test_e4m3_rn_against_torch(oracle_mod):
    rng = np.random.default_rng(3)
    ss = np.exp(rng.uniform(math.log(1e-4), math.log(440), 6000)).astype(np.float32)
    # exact midpoints between neighbouring codes (ties)
    vals = [float(v) for _, v in bounds.E4M3]
    mids = np.array([(a + b) / 2 for a, b in zip(vals, vals[1:])], dtype=np.float64).astype(np.float32)
    allv = np.concatenate([ss, mids])
    tq = torch.from_numpy(allv).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    for s, c in zip(allv, tq):
        assert oracle_mod.e4m3_rn(float(s)) == int(c), s
    assert oracle_mod.e4m3_rn(1e6) == 126  # saturates to 448
    assert oracle_mod.e4m3_rn(0.0) == 0
