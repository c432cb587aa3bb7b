"""Invariants that pin the oracle's sweep, baselines, scales and layouts.

Each test checks the oracle against something other than itself: an
independent exact-rational re-implementation, a property the paper proves
(Lemmas 4.1-4.3, the Appendix-C optimum as a lower bound, ScaleSweep's window
containing the AbsMax and 4/6 codes), a closed form, or a library routine.
"""
import math
from fractions import Fraction

import numpy as np
import pytest
import torch

from oracle import bounds
from paper_2606_07618_gb300 import workloads as W

GRID = [Fraction(g) for g in (0, 0.5, 1, 1.5, 2, 3, 4, 6)]


def _f32(t):
    return t.float().numpy() if isinstance(t, torch.Tensor) else np.asarray(t, np.float32)


# --------------------------------------------------------------------------- brute force
def _rne_mag(t):
    a = abs(Fraction(float(t)))
    d = [abs(a - g) for g in GRID]
    m = min(d)
    ks = [k for k in range(8) if d[k] == m]
    k = ks[0] if len(ks) == 1 else [k for k in ks if k % 2 == 0][0]
    return GRID[k], k


def _brute_block(x, S, w=None, lo=-126, hi=126):
    """Independent exact re-implementation of one block's sweep: float32 for
    the decisions (numpy IEEE ops), exact rationals for the loss."""
    S = np.float32(S)
    E = np.float32(1) / S
    y = (np.asarray(x, np.float32) * E).astype(np.float32)
    m = np.max(np.abs(y))
    sbase = np.float32(m) / np.float32(6)
    I0 = max([c for c, v in bounds.E4M3 if v <= Fraction(float(sbase))])
    clo, chi = min(max(I0 + lo, 1), 126), min(max(I0 + hi, 1), 126)
    _brute_block.window = (clo, chi)
    best, bestc, bestq = None, None, None
    for c in range(clo, chi + 1):
        v = bounds.E4M3[c][1]
        r = np.float32(1) / np.float32(float(v))
        L = Fraction(0)
        qs = []
        for i, yi in enumerate(y):
            t = np.float32(yi * r)
            g, k = _rne_mag(t)
            qs.append((8 if math.copysign(1.0, float(t)) < 0 else 0) | k)
            wi = Fraction(float(w[i])) if w is not None else Fraction(1)
            e = Fraction(float(yi)) - (g if t >= 0 else -g) * v
            L += wi * e * e
        if best is None or L < best:
            best, bestc, bestq = L, c, qs
    return bestc, best, bestq


def test_bruteforce_matches_oracle_small_blocks(oracle_mod):
    rng = np.random.default_rng(11)
    for trial in range(60):
        dist = trial % 3
        if dist == 0:
            x = rng.standard_normal(16) * 0.02
        elif dist == 1:
            x = rng.standard_t(3, 16)
        else:
            x = rng.laplace(0, 0.015, 16)
            x[rng.integers(16)] *= 30
        x = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).float().numpy().reshape(1, 16)
        S = np.float32(np.max(np.abs(x))) / np.float32(1536)
        w = np.exp(rng.standard_normal(16)).astype(np.float32) if trial % 2 else None
        obj = oracle_mod.WMSE if w is not None else oracle_mod.MSE
        for lo, hi in ((-126, 126), oracle_mod.default_window(obj, 16)):
            bc, bL, bq = _brute_block(x[0], S, w, lo, hi)
            o = oracle_mod.quantize(0, x, 16, float(S), obj, w=w, w_row_stride=0, window=(lo, hi),
                                    want_cand=True, cand_stride=128)
            clo, chi = _brute_block.window
            assert int(o["cand_lo"][0]) == clo
            assert int(np.count_nonzero(~np.isnan(o["cand"][0]))) == chi - clo + 1
            assert int(o["sf"][0, 0]) == bc
            assert abs(o["best"][0] - float(bL)) <= 1e-12 * float(bL) + 1e-300
            packed = [(o["codes"][0, j // 2] >> (4 * (j % 2))) & 0xF for j in range(16)]
            assert packed == bq


# Blocks built on multiples of an edge candidate's value (S = 1): the
# exhaustive optimum sits exactly on the window edge, so the window's ends are
# exercised.  MSE: optimum at I0+7 (Lemma 4.2's bound is attained).  WMSE:
# optimum at I0-8 (the empirical s_base/2 bound of Sec. 4.2.2 is attained).
EDGE_BLOCKS = [
    (0, 7, [-6.75, -4.5, 1.125, -4.5, 2.25] + [0.0] * 10 + [7.9917088], None),
    (1, -8, [0.375, 1.5, 1.5, -1.125, -1.5, 1.125, -1.5, 3.0, -3.0, 2.25, 0, 0, 0, 0, 0, 9.607283],
     [1.4044138, 1.5277122, 1.4495127, 1.466322, 1.3763213, 0.6984349, 0.14932422, 0.8968069, 0.44765526,
      2.9451609, 0.7491871, 1.0870584, 0.4275834, 0.6001219, 0.9885332, 0.0039137434]),
]


def test_window_edge_blocks(oracle_mod):
    for obj, offset, yv, wv in EDGE_BLOCKS:
        y = np.array(yv, np.float32).reshape(1, 16)
        w = None if wv is None else np.array(wv, np.float32)
        bc, bL, bq = _brute_block(y[0], 1.0, w, -126, 126)
        I0 = oracle_mod.e4m3_floor(float(np.float32(np.abs(y).max()) / np.float32(6)))
        assert bc - I0 == offset
        o = oracle_mod.quantize(0, y, 16, 1.0, obj, w=w)
        assert int(o["sf"][0, 0]) == bc
        assert abs(o["best"][0] - float(bL)) <= 1e-12 * float(bL)


# --------------------------------------------------------------------------- Lemma 4.3 / window
@pytest.fixture(scope="module")
def weight2048():
    t = W.workload("weight-2048").tensors[0]
    return _f32(W.draw(t))


def test_bounded_equals_exhaustive_weight2048(oracle_mod, weight2048):
    """Sec. 4.2.2: the [-3, 7] MSE window holds the exhaustive optimum
    (Lemma 4.3 for blocks with (11/7) s_base^FP8 <= 448, Lemma 4.1/4.2 on top).
    Checked on every block of the 2048x2048 N(0, 0.02^2) matrix, D = 448."""
    x = weight2048
    S, _ = oracle_mod.global_scale(x, 448.0)
    b = oracle_mod.quantize(0, x, 16, S, oracle_mod.MSE)
    e = oracle_mod.quantize(0, x, 16, S, oracle_mod.MSE, window=(-126, 126))
    assert np.array_equal(b["best"], e["best"])
    assert np.array_equal(b["sf"], e["sf"])
    assert np.array_equal(b["codes"], e["codes"])


def test_wmse_window_vs_exhaustive_reported(oracle_mod, weight2048):
    """The WMSE lower bound s_base/2 is empirical (Sec. 4.2.2); report misses,
    require them to be rare."""
    x = weight2048[:512]
    w = np.exp(np.random.default_rng(5).standard_normal(x.shape[1])).astype(np.float32)
    S, _ = oracle_mod.global_scale(x, 256.0)
    b = oracle_mod.quantize(0, x, 16, S, oracle_mod.WMSE, w=w)
    e = oracle_mod.quantize(0, x, 16, S, oracle_mod.WMSE, w=w, window=(-126, 126))
    miss = np.mean(b["best"] > e["best"])
    print(f"WMSE [-8,7] misses the exhaustive optimum on {miss:.2e} of blocks")
    assert miss < 1e-3
    assert np.all(b["best"] >= e["best"])


def _mixed_inputs(rows=96, cols=256, seed=3):
    out = []
    for i, dist in enumerate(["normal", "student_t", "laplace"]):
        std = {"normal": 0.02, "student_t": 1.0, "laplace": 0.015}[dist]
        out.append(_f32(W.small_tensor(rows, cols, seed + i, dist=dist, std=std, outliers=3, mult=30.0)))
    return out


@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("objective", [0, 1])
def test_scalesweep_dominates_absmax_and_four_six(oracle_mod, block, objective):
    """AbsMax's code lies in {I0, I0+1} and the 4/6 code lies at most I0+7
    (Lemma 4.2 with alpha = 3/2, plus one for rounding up), so the sweep's
    optimum can be no worse than either under the same S and objective."""
    for x in _mixed_inputs():
        S, _ = oracle_mod.global_scale(x, 256.0)
        w = np.exp(np.random.default_rng(9).standard_normal(x.shape[1])).astype(np.float32) if objective else None
        ss = oracle_mod.quantize(0, x, block, S, objective, w=w)
        am = oracle_mod.quantize(1, x, block, S, objective, w=w)
        fs = oracle_mod.quantize(2, x, block, S, objective, w=w)
        assert np.all(ss["best"] <= am["best"])
        assert np.all(ss["best"] <= fs["best"])
        assert np.all(fs["best"] <= am["best"])
        # the recorded AbsMax loss is the loss of its own scale codes
        Lam = oracle_mod.block_losses_at(x, block, S, am["sf"], objective, w=w)
        assert np.array_equal(Lam, am["best"])
        Lss, css = oracle_mod.block_losses_at(x, block, S, ss["sf"], objective, w=w, want_codes=True)
        assert np.array_equal(Lss, ss["best"]) and np.array_equal(css, ss["codes"])


def test_lemma1_halving_in_oracle_arithmetic(oracle_mod):
    """Lemma 4.1 on the oracle's own per-candidate losses: for every window
    candidate with v_c > m/3.5 whose half is also evaluated, L(v_c/2) <= L(v_c)."""
    x = _mixed_inputs(64, 256, 21)[0]
    S, _ = oracle_mod.global_scale(x, 256.0)
    o = oracle_mod.quantize(0, x, 16, S, oracle_mod.WMSE, w=np.ones(x.shape[1], np.float32), want_cand=True)
    E = np.float32(1) / np.float32(S)
    y = (x * E).astype(np.float32).reshape(-1, 16)
    m = np.abs(y).max(axis=1)
    checked = 0
    for b in range(y.shape[0]):
        lo = o["cand_lo"][b]
        for k in range(16):
            c = lo + k
            if c > 126 or np.isnan(o["cand"][b, k]) or c - 8 < lo or c < 16:
                continue
            if oracle_mod.e4m3_value(c) * 3.5 > m[b]:
                assert o["cand"][b, k - 8] <= o["cand"][b, k] * (1 + 1e-9)
                checked += 1
    assert checked > 100


# --------------------------------------------------------------------------- Appendix C
def _loss_np(y, w, s):
    a = np.abs(y.astype(np.float64))
    g = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6])
    q = g[np.argmin(np.abs(a[:, None] / s - g[None, :]), axis=1)]
    return float(np.sum((w if w is not None else 1.0) * (a - s * q) ** 2))


def test_opt_scale_against_dense_scan(oracle_mod):
    rng = np.random.default_rng(4)
    for trial in range(40):
        n = [1, 2, 4, 16][trial % 4]
        y = (rng.standard_normal(n) * 3).astype(np.float32)
        w = np.exp(rng.standard_normal(n)).astype(np.float32) if trial % 2 else None
        s_opt, L_opt = oracle_mod.opt_scale(y, w)
        assert abs(_loss_np(y, w, s_opt) - L_opt) <= 1e-9 * (1 + L_opt)
        m = float(np.max(np.abs(y)))
        for s in np.geomspace(m / 12, m * 8, 3000):
            assert _loss_np(y, w, s) >= L_opt * (1 - 1e-12) - 1e-15
    s_opt, L_opt = oracle_mod.opt_scale(np.array([0, 0, 3.3, 0], np.float32))
    assert L_opt == 0.0


def test_optimal_fp32_scale_lower_bounds_every_fp8_result(oracle_mod):
    rng = np.random.default_rng(8)
    for x in _mixed_inputs(24, 256, 31):
        S, _ = oracle_mod.global_scale(x, 256.0)
        E = np.float32(1) / np.float32(S)
        for objective in (0, 1):
            w = np.exp(rng.standard_normal(x.shape[1])).astype(np.float32) if objective else None
            ss = oracle_mod.quantize(0, x, 16, S, objective, w=w)
            am = oracle_mod.quantize(1, x, 16, S, objective, w=w)
            y = (x * E).astype(np.float32).reshape(x.shape[0], -1, 16)
            for r in range(0, x.shape[0], 3):
                for k in range(y.shape[1]):
                    b = r * y.shape[1] + k
                    wb = w[16 * k:16 * k + 16] if w is not None else None
                    s_opt, L_opt = oracle_mod.opt_scale(y[r, k], wb)
                    assert L_opt <= ss["best"][b] * (1 + 1e-12) + 1e-300
                    assert L_opt <= am["best"][b] * (1 + 1e-12) + 1e-300
                    if objective == 0:
                        _, L8 = oracle_mod.fp8_opt_code(y[r, k], wb, s_opt)
                        assert ss["best"][b] <= L8 * (1 + 1e-12)


def _exact_loss_at(y, w, c):
    """Exact-rational loss of scale code c on the float32 block y, with the
    float32 rounding decisions of the contract (independent of the oracle)."""
    v = bounds.E4M3[c][1]
    r = np.float32(1) / np.float32(float(v))
    L = Fraction(0)
    for i, yi in enumerate(np.asarray(y, np.float32)):
        t = np.float32(yi * r)
        g, _ = _rne_mag(t)
        wi = Fraction(float(w[i])) if w is not None else Fraction(1)
        e = Fraction(float(yi)) - (g if t >= 0 else -g) * v
        L += wi * e * e
    return L


def _floor_ceil_codes(s):
    """floor_E4M3 / ceil_E4M3 of a positive real s as codes in 1..126, from the
    exact value table (floor clamped up to code 1, ceil down to code 126)."""
    sf = Fraction(s)
    fl = max([c for c, v in bounds.E4M3 if c >= 1 and v <= sf], default=1)
    ce = min([c for c, v in bounds.E4M3 if c >= 1 and v >= sf], default=126)
    return fl, ce


def test_fp8_quantised_optimum_picks_better_of_floor_and_ceil(oracle_mod):
    """Appendix C's FP8-quantised optimum: of floor_E4M3(s*) and ceil_E4M3(s*)
    the one with the lower loss, ties to the floor.  Checked against the exact
    E4M3 table and exact-rational losses on sampled blocks of every
    distribution, then on three constructed blocks where the ceiling is
    strictly better, the floor is strictly better, and the two tie."""
    rng = np.random.default_rng(12)
    picked = {"floor": 0, "ceil": 0, "same": 0}
    for x in _mixed_inputs(8, 128, 91):
        S, _ = oracle_mod.global_scale(x, 256.0)
        E = np.float32(1) / np.float32(S)
        y = (x * E).astype(np.float32).reshape(-1, 16)
        for b in rng.choice(y.shape[0], 12, replace=False):
            for objective in (0, 1):
                w = np.exp(rng.standard_normal(16)).astype(np.float32) if objective else None
                s_opt, _ = oracle_mod.opt_scale(y[b], w)
                code, L = oracle_mod.fp8_opt_code(y[b], w, s_opt)
                fl, ce = _floor_ceil_codes(s_opt)
                Lf, Lc = _exact_loss_at(y[b], w, fl), _exact_loss_at(y[b], w, ce)
                want = ce if Lc < Lf else fl
                picked["same" if fl == ce else ("ceil" if want == ce else "floor")] += 1
                assert code == want, (b, objective, fl, ce, float(Lf), float(Lc))
                assert abs(L - float(min(Lf, Lc))) <= 1e-12 * float(min(Lf, Lc)) + 1e-300
    assert picked["floor"] > 0 and picked["ceil"] > 0
    # constructed: s* = 1.05 lies between code 56 (1.0) and code 57 (1.125)
    spike = np.zeros(16, np.float32)
    spike[3] = 6.75                              # 6 * 1.125: exact at the ceiling, 0.75 off at the floor
    assert oracle_mod.fp8_opt_code(spike, None, 1.05) == (57, 0.0)
    spike[3] = 6.0                               # exact at the floor, 0.75 off at the ceiling
    assert oracle_mod.fp8_opt_code(spike, None, 1.05) == (56, 0.0)
    spike[3] = 1e-3                              # rounds to 0 under both: equal losses -> the floor
    code, L = oracle_mod.fp8_opt_code(spike, None, 1.05)
    assert code == 56 and L == float(np.float32(1e-3)) ** 2
    # s* on a code, below the smallest code and above the largest
    assert oracle_mod.fp8_opt_code(spike, None, 1.0)[0] == 56
    assert oracle_mod.fp8_opt_code(spike, None, 2.0 ** -11)[0] == 1
    assert oracle_mod.fp8_opt_code(spike, None, 500.0)[0] == 126


# --------------------------------------------------------------------------- closed forms
def test_single_spike_block(oracle_mod):
    for code, sign in ((58, 1.0), (58, -1.0), (40, 1.0), (90, -1.0)):
        v = oracle_mod.e4m3_value(code)
        x = np.zeros((1, 16), np.float32)
        x[0, 5] = sign * 6 * v
        o = oracle_mod.quantize(0, x, 16, 1.0, oracle_mod.MSE)
        assert o["best"][0] == 0.0
        assert o["sf"][0, 0] == code          # lowest code that represents the spike
        nib = (o["codes"][0, 2] >> 4) & 0xF
        assert nib == (0xF if sign < 0 else 0x7)
        rest = [(o["codes"][0, j // 2] >> (4 * (j % 2))) & 0xF for j in range(16) if j != 5]
        assert all(q == 0 for q in rest)


def test_power_of_two_rescaling_invariance(oracle_mod):
    x = _mixed_inputs(32, 128, 41)[2]
    S, _ = oracle_mod.global_scale(x, 256.0)
    ref = oracle_mod.quantize(0, x, 16, S, oracle_mod.MSE)
    for k in (-3, 5):
        xs = (x * np.float32(2.0 ** k)).astype(np.float32)
        Sk, _ = oracle_mod.global_scale(xs, 256.0)
        assert Sk == np.float32(S) * np.float32(2.0 ** k)
        o = oracle_mod.quantize(0, xs, 16, Sk, oracle_mod.MSE)
        assert np.array_equal(o["codes"], ref["codes"]) and np.array_equal(o["sf"], ref["sf"])


def test_wmse_with_unit_weights_is_mse(oracle_mod):
    x = _mixed_inputs(32, 128, 51)[1]
    S, _ = oracle_mod.global_scale(x, 256.0)
    a = oracle_mod.quantize(0, x, 16, S, oracle_mod.MSE, window=(-8, 7))
    b = oracle_mod.quantize(0, x, 16, S, oracle_mod.WMSE, w=np.ones(128, np.float32), window=(-8, 7))
    assert np.array_equal(a["codes"], b["codes"]) and np.array_equal(a["sf"], b["sf"])
    assert np.array_equal(a["best"], b["best"])


def test_zero_blocks_and_zero_tensor(oracle_mod):
    x = _mixed_inputs(4, 64, 61)[0].copy()
    x[1, 16:32] = 0.0
    x[1, 20] = -0.0
    S, _ = oracle_mod.global_scale(x, 256.0)
    o = oracle_mod.quantize(0, x, 16, S, oracle_mod.MSE)
    assert o["sf"][1, 1] == 0
    nibs = [(o["codes"][1, 8 + j // 2] >> (4 * (j % 2))) & 0xF for j in range(16)]
    assert nibs == [8 if j == 4 else 0 for j in range(16)]
    z = np.zeros((2, 32), np.float32)
    z[0, 3] = -0.0
    Sz, bad = oracle_mod.global_scale(z, 256.0)
    assert Sz == 0.0 and not bad
    o = oracle_mod.quantize(0, z, 16, Sz, oracle_mod.MSE)
    assert np.all(o["sf"] == 0)
    assert o["codes"][0, 1] == 0x80 and np.count_nonzero(o["codes"]) == 1


def test_nonfinite_and_out_of_range_blocks(oracle_mod):
    """Zero rule for non-finite and out-of-range blocks (a reading: the paper
    defines no output for them).  Every other block must come out exactly as
    in the clean tensor (blocks are independent given S, Sec. 4.2.1), and a
    block just below the 2^48 bound is swept normally -- the exact-rational
    brute force agrees with it."""
    x = _mixed_inputs(4, 64, 71)[1].copy()
    S, _ = oracle_mod.global_scale(x, 256.0)
    Sf = np.float32(S)
    E = np.float32(1) / Sf
    xp = x.copy()
    xp[0, 16 + 5] = np.nan
    xp[1, 7] = np.inf
    xp[2, 32 + 2] = -np.inf
    xp[2, 32 + 3] = -0.0
    big = np.float32(2.0 ** 48)
    xp[3, 16 + 9] = np.float32(big / E)          # y = fl(x E) lands on or above 2^48
    while np.float32(xp[3, 16 + 9] * E) < big:
        xp[3, 16 + 9] = np.nextafter(xp[3, 16 + 9], np.float32(np.inf))
    xp[3, 48 + 4] = np.float32(2.0 ** 47 / E)    # y around 2^47: swept normally
    planted = {(0, 1), (1, 0), (2, 2), (3, 1)}
    y_planted = (xp * E).astype(np.float32)
    for method in (0, 1, 2):
        for objective in (0, 1):
            w = np.exp(np.random.default_rng(3).standard_normal(64)).astype(np.float32) if objective else None
            ref = oracle_mod.quantize(method, x, 16, S, objective, w=w)
            got = oracle_mod.quantize(method, xp, 16, S, objective, w=w)
            for r in range(4):
                for k in range(4):
                    nib = [(got["codes"][r, 8 * k + j // 2] >> (4 * (j % 2))) & 0xF for j in range(16)]
                    if (r, k) in planted:
                        assert got["sf"][r, k] == 0, (method, objective, r, k)
                        want = [8 if math.copysign(1.0, float(v)) < 0 else 0 for v in y_planted[r, 16 * k:16 * k + 16]]
                        assert nib == want, (method, objective, r, k)
                    elif (r, k) != (3, 3):
                        assert got["sf"][r, k] == ref["sf"][r, k]
                        assert np.array_equal(got["codes"][r, 8 * k:8 * k + 8], ref["codes"][r, 8 * k:8 * k + 8])
            # the 2^47 block is an ordinary block: saturating scales, no zero rule
            assert got["sf"][3, 3] >= 119
            if method == 0:
                wb = None if w is None else w[48:64]
                bc, _, bq = _brute_block(xp[3, 48:64], S, wb, *oracle_mod.default_window(objective, 16))
                assert got["sf"][3, 3] == bc
                nib = [(got["codes"][3, 24 + j // 2] >> (4 * (j % 2))) & 0xF for j in range(16)]
                assert nib == bq


def test_global_scale_planted_max(oracle_mod):
    rng = np.random.default_rng(12)
    x = rng.uniform(-1, 1, 100003).astype(np.float32)
    x[777] = -3.75
    for D in (448.0, 256.0):
        S, bad = oracle_mod.global_scale(x, D)
        assert S == np.float32(3.75) / np.float32(6 * D) and not bad
    x2 = x.copy()
    x2[5] = np.nan
    S, bad = oracle_mod.global_scale(x2, 256.0)
    assert bad and S == np.float32(3.75) / np.float32(1536)
    x2[6] = -np.inf
    S, bad = oracle_mod.global_scale(x2, 256.0)
    assert bad and math.isinf(S)


def test_dequantize_matches_format_tables(oracle_mod):
    rng = np.random.default_rng(13)
    rows, cols, block = 37, 96, 16
    codes = rng.integers(0, 256, (rows, cols // 2), dtype=np.uint8)
    sf = rng.integers(0, 127, (rows, cols // block), dtype=np.uint8)
    S = np.float32(0.0123)
    grid = np.array([0, 0.5, 1, 1.5, 2, 3, 4, 6, -0.0, -0.5, -1, -1.5, -2, -3, -4, -6], np.float32)
    v = torch.from_numpy(sf).view(torch.float8_e4m3fn).float().numpy()
    q = np.empty((rows, cols), np.float32)
    q[:, 0::2] = grid[codes & 0xF]
    q[:, 1::2] = grid[codes >> 4]
    want = ((q * np.repeat(v, block, axis=1)).astype(np.float32) * S).astype(np.float32)
    got = oracle_mod.dequantize(codes, sf, oracle_mod.LAYOUT_LINEAR, float(S), rows, cols, block)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    got16 = oracle_mod.dequantize(codes, sf, oracle_mod.LAYOUT_LINEAR, float(S), rows, cols, block, out_bf16=True)
    want16 = torch.from_numpy(want).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got16, want16)
    swz = oracle_mod.swizzle_scales(sf)
    got_s = oracle_mod.dequantize(codes, swz, oracle_mod.LAYOUT_SWIZZLED, float(S), rows, cols, block)
    assert np.array_equal(got_s.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("rows,kb", [(1, 1), (130, 5), (128, 4), (256, 8), (300, 13)])
def test_swizzle_layout_structure(oracle_mod, rows, kb):
    """Structural checks of the swizzled layout on CPU (the layout itself is
    pinned against cuBLASLt in test_gpu_swizzle_pin.py): a bijection into the
    padded buffer, zero pads, 512-byte 128x4 atoms, rows r, r+32, r+64, r+96
    sharing one 16-byte line."""
    nbytes = oracle_mod.swizzle_bytes(rows, kb)
    assert nbytes == -(-rows // 128) * 128 * (-(-kb // 4)) * 4
    offs = {oracle_mod.swizzle_offset(r, k, kb) for r in range(rows) for k in range(kb)}
    assert len(offs) == rows * kb and max(offs) < nbytes
    sf = (np.arange(rows * kb) % 126 + 1).astype(np.uint8).reshape(rows, kb)
    out = oracle_mod.swizzle_scales(sf)
    assert np.count_nonzero(out) == rows * kb
    if rows >= 128 and kb >= 4:
        for r in range(32):
            base = oracle_mod.swizzle_offset(r, 0, kb)
            assert base == r * 16
            assert [oracle_mod.swizzle_offset(r + 32 * j, k, kb) for j in range(4) for k in range(4)] == \
                list(range(base, base + 16))


def test_absmax_and_four_six_scales_use_rn(oracle_mod):
    """Sec. 3.2: s_k = RN_FP8(blockmax / (6 S)); 4/6 also tries RN_FP8(blockmax / (4 S))
    and keeps the lower loss.  RN is taken from torch's float8_e4m3fn cast."""
    for x in _mixed_inputs(16, 128, 71):
        S, _ = oracle_mod.global_scale(x, 256.0)
        E = np.float32(1) / np.float32(S)
        y = (x * E).astype(np.float32).reshape(-1, 16)
        m = np.abs(y).max(axis=1).astype(np.float32)
        rn6 = torch.from_numpy((m / np.float32(6)).astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8)
        rn4 = torch.from_numpy((m / np.float32(4)).astype(np.float32)).to(torch.float8_e4m3fn).view(torch.uint8)
        c6 = np.maximum(rn6.numpy(), 1)
        c4 = np.maximum(rn4.numpy(), 1)
        am = oracle_mod.quantize(1, x, 16, S, oracle_mod.MSE)
        assert np.array_equal(am["sf"].reshape(-1), c6)
        fs = oracle_mod.quantize(2, x, 16, S, oracle_mod.MSE)
        L6 = oracle_mod.block_losses_at(x, 16, S, c6)
        L4 = oracle_mod.block_losses_at(x, 16, S, c4)
        want = np.where(L4 < L6, c4, c6)
        assert np.array_equal(fs["sf"].reshape(-1), want)
        # the two losses 4/6 compares are exactly L(c4) and L(c6)
        assert np.array_equal(np.minimum(fs["best"], fs["second"]), np.minimum(L4, L6))
        assert np.array_equal(np.maximum(fs["best"], fs["second"]), np.maximum(L4, L6))
