"""Pins of the per-block tight window (NVFP4_WINDOW_TIGHT) on the CPU.

The tight window keeps the default window's argmin (lowest code on ties) while
dropping candidates the paper proves useless, block by block:
* upper end: every code c >= 16 with 3.5 v_c > max|y| goes (Lemma 4.1: such a
  scale never beats half of it, which is code c - 8 and stays in the window;
  below 16 half a scale need not be a code -- subnormal code 3 has no half);
* lower end, MSE with 16-element blocks: the per-mantissa bound of Table 2 /
  Lemma 4.3, I0 - delta(b) with delta from the exact rational table in
  oracle/bounds.py (not from the kernel's constants), for I0 in 16..120.
Checked on the oracle's float64 candidate losses: the argmin over each block's
tight window equals the oracle's choice over the full default window, on
several distributions and global scales, both objectives, blocks 16/32/64.  A
planted mistake (the cut applied to the subnormal codes, or compared with
s_base instead of max|y|) must break it.
"""
import numpy as np
import pytest

import oracle
from oracle import bounds

DELTA = {b: d for b, _, d in bounds.lower_table()}


def block_stats(x, S, block):
    """m = max|fl32(x * fl32(1/S))| and I0 = floor_E4M3(fl32(m / 6)) per block."""
    E = np.float32(1.0) / np.float32(S)
    y = (x.astype(np.float32) * E).astype(np.float32)
    m = np.abs(y).reshape(-1, block).max(axis=1)
    sb = (m / np.float32(6.0)).astype(np.float32)
    I0 = np.array([oracle.e4m3_floor(float(v)) for v in sb], dtype=np.int64)
    return m.astype(np.float64), I0


def tight_windows(m, I0, objective, block, lower=None, cut=3.5, cut_from=16):
    v = np.array([oracle.e4m3_value(c) for c in range(127)])
    lo_def = -3 if (objective == oracle.MSE and block == 16) else -8
    clo = np.empty_like(I0)
    chi = np.empty_like(I0)
    for k, (mk, i0) in enumerate(zip(m, I0)):
        lo = lo_def
        if objective == oracle.MSE and block == 16 and 16 <= i0 <= 120:
            lo = -(lower or DELTA)[int(i0) & 7]
        a = min(max(i0 + lo, 1), 126)
        b = min(max(i0 + 7, 1), 126)
        while b > a and b >= cut_from and cut * v[b] > mk:   # half of v_b is code b - 8 from 16 up
            b -= 1
        clo[k], chi[k] = a, b
    return clo, chi


def tight_choice(ref, clo, chi):
    """Lowest-code argmin of the oracle's candidate losses restricted to [clo, chi]."""
    cand, lo = ref["cand"], ref["cand_lo"].astype(np.int64)
    out = np.empty(len(lo), dtype=np.int64)
    for k in range(len(lo)):
        a, b = clo[k] - lo[k], chi[k] - lo[k]
        seg = cand[k, a:b + 1]
        out[k] = lo[k] + a + int(np.argmin(seg))          # argmin returns the first (lowest) minimum
    return out


def make(dist, rows, cols, seed):
    rng = np.random.default_rng(seed)
    if dist == "normal":
        x = rng.standard_normal((rows, cols)) * 0.02
    elif dist == "student_t":
        x = rng.standard_t(3, (rows, cols))
    else:
        x = rng.laplace(0.0, 0.015, (rows, cols))
    x[:, rng.integers(0, cols, 2)] *= 30.0
    return x.astype(np.float32)


@pytest.mark.parametrize("objective,block", [(oracle.MSE, 16), (oracle.WMSE, 16), (oracle.MSE, 32),
                                             (oracle.WMSE, 64)])
@pytest.mark.parametrize("dist", ["normal", "student_t", "laplace"])
def test_tight_window_keeps_the_argmin(objective, block, dist):
    x = make(dist, 96, 256, {"normal": 11, "student_t": 12, "laplace": 13}[dist] * block)
    w = np.exp(np.random.default_rng(1).standard_normal(256)).astype(np.float32) if objective else None
    for D in (256.0, 448.0, 0.05):                   # 448: I0 = 126 at the top; 0.05: I0 below 16
        S, _ = oracle.global_scale(x, D)
        ref = oracle.quantize(0, x, block, S, objective, w=w, want_cand=True)
        m, I0 = block_stats(x, S, block)
        clo, chi = tight_windows(m, I0, objective, block)
        live = m > 0
        assert np.all(clo[live] <= chi[live])
        got = tight_choice(ref, clo, chi)
        assert np.array_equal(got[live], ref["sf"].reshape(-1)[live].astype(np.int64))


def test_tight_window_prunes_and_planted_mistakes_are_caught():
    x = make("normal", 256, 256, 5)
    S, _ = oracle.global_scale(x, 256.0)
    ref = oracle.quantize(0, x, 16, S, oracle.MSE, want_cand=True)
    m, I0 = block_stats(x, S, 16)
    clo, chi = tight_windows(m, I0, oracle.MSE, 16)
    width = chi - clo + 1
    assert width.mean() < 10.0 and width.max() <= 11      # it does prune, never widens
    want = ref["sf"].reshape(-1).astype(np.int64)
    # planted mistakes each lose real minimizers: the cut compared with s_base
    # = m/6 instead of m, and (at small scales) the cut applied below code 16
    clo2, chi2 = tight_windows(m, I0, oracle.MSE, 16, cut=3.5 * 6)
    assert not np.array_equal(tight_choice(ref, clo2, chi2), want)
    S2, _ = oracle.global_scale(x, 0.05)
    ref2 = oracle.quantize(0, x, 16, S2, oracle.MSE, want_cand=True)
    m2, I02 = block_stats(x, S2, 16)
    live = m2 > 0
    clo2, chi2 = tight_windows(m2, I02, oracle.MSE, 16, cut_from=1)
    assert not np.array_equal(tight_choice(ref2, clo2, chi2)[live], ref2["sf"].reshape(-1)[live].astype(np.int64))
    # the lower end is tightened where it applies (Table 2 itself is pinned
    # against the paper's printed table in test_oracle_bounds.py; no sampled block
    # sits at it, so a bound one code too high cannot be caught by results)
    rng16 = (I0 >= 16) & (I0 <= 120)
    assert np.all(clo[rng16] >= I0[rng16] - 3) and np.mean(clo[rng16] == I0[rng16] - 2) > 0.5
