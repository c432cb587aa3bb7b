"""The sweep's warp-uniform offset bound is sound in fp32.

The default-window sweeps skip a candidate scale when, for every lane of a warp,
a lower bound on the block's loss exceeds the lane's best loss so far.  The
bound is the error terms of the largest |y| of each half of a lane's
16-element segment, summed over the block's lanes and multiplied by 1 - 2^-20;
the claim is that the candidate's loss, as the kernels compute it in fp32
(errors e = fl(y - q v) from q = RNE_E2M1(fl(y fl(1/v))), weighted products
accumulated by fused multiply-adds into two interleaved running sums per lane,
the two sums added, then the lanes' losses added pairwise), is never below that
bound.  This test computes both sides on the CPU the way the kernels order and
round them (float32 results of float64 operations on float32 inputs: the
products are exact there, so each step is one rounding, up to the rare double
rounding of a fused multiply-add's sum, far inside the 2^-20 margin) over blocks
of 16, 32 and 64 drawn to stress the bound -- heavy tails, repeated maxima,
near-ties between halves, tiny and huge magnitudes, zero weights -- and over
every candidate of the window, including those the bound is meant to skip.
"""
import numpy as np
import pytest

F32, F64 = np.float32, np.float64
GRID = np.array([0.0, 0.5, 1.0, 1.5, 2.0, 3.0, 4.0, 6.0])
MARGIN = F32(1.0 - 2.0 ** -20)


def e4m3_value(c):
    e, m = c >> 3, c & 7
    return (m / 8.0) * 2.0 ** -6 if e == 0 else (1.0 + m / 8.0) * 2.0 ** (e - 7)


def f32(x):
    return np.asarray(x, dtype=F64).astype(F32)


def rne_e2m1(t):
    """Nearest E2M1 magnitude, ties to the even code, saturating at 6."""
    a = np.minimum(np.abs(t.astype(F64)), 6.0)
    d = np.abs(a[..., None] - GRID)
    best = d.min(-1, keepdims=True)
    cand = np.where(d == best, np.arange(8), 99)
    # among tied grid points take the even code (codes 0..7 in grid order)
    idx = np.where(np.any((cand % 2 == 0) & (cand < 99), -1), np.min(np.where(cand % 2 == 0, cand, 99), -1),
                   np.min(cand, -1))
    return GRID[idx] * np.sign(t)


def cand_err(y, v):
    """e = fl(y - q v) with q = RNE_E2M1(fl(y * fl(1/v))), as cand_err2."""
    r = f32(1.0 / v)
    t = f32(y.astype(F64) * F64(r))
    q = rne_e2m1(t)
    return f32(y.astype(F64) - q * v)


def lane_loss(y, w, v, wmse):
    """One lane's loss: terms of elements 2j into the low sum, 2j+1 into the
    high sum, j ascending (fma: exact product plus accumulator, one rounding),
    then the two sums added."""
    e = cand_err(y, v)
    we = f32(w.astype(F64) * e.astype(F64)) if wmse else e
    acc = np.zeros(y.shape[:-1] + (2,), dtype=F32)
    for j in range(8):
        for h in range(2):
            k = 2 * j + h
            acc[..., h] = f32(we[..., k].astype(F64) * e[..., k].astype(F64) + acc[..., h].astype(F64))
    return f32(acc[..., 0].astype(F64) + acc[..., 1].astype(F64))


def lane_bound(y, w, v, wmse):
    """The two terms of the largest |y| of each half, added (per lane)."""
    ay = np.abs(y)
    out = []
    for h in range(2):
        part = ay[..., 8 * h:8 * h + 8]
        m = part.max(-1)
        if wmse:   # the weight of the last element of the half at its maximum, as the kernel selects it
            at = part == m[..., None]
            idx = 7 - np.argmax(at[..., ::-1], -1)
            wm = np.take_along_axis(w[..., 8 * h:8 * h + 8], idx[..., None], -1)[..., 0]
        e = cand_err(m.astype(F32), v)
        t = f32(f32(wm.astype(F64) * e) * e.astype(F64)) if wmse else f32(e.astype(F64) * e.astype(F64))
        out.append(t)
    return f32(out[0].astype(F64) + out[1].astype(F64))


def group_sum(x, segs):
    """xor-shuffle sums over the block's lanes (last axis = lanes)."""
    if segs >= 2:
        x = f32(x.astype(F64) + x[..., [1, 0] + ([3, 2] if segs == 4 else [])].astype(F64))
    if segs >= 4:
        x = f32(x.astype(F64) + x[..., [2, 3, 0, 1]].astype(F64))
    return x[..., 0]


def blocks(kind, n, block, rng):
    if kind == "laplace":
        y = rng.laplace(0.0, 1.0, (n, block))
    elif kind == "student_t":
        y = rng.standard_t(3, (n, block))
    elif kind == "normal":
        y = rng.standard_normal((n, block))
    elif kind == "repeated_max":          # the maximum appears in both halves, with both signs
        y = rng.standard_normal((n, block))
        y[:, 8] = -np.abs(y).max(-1)
        y[:, 0] = np.abs(y).max(-1)
    else:                                 # "spiky": one or two dominant elements, the rest tiny
        y = rng.standard_normal((n, block)) * 1e-3
        y[np.arange(n), rng.integers(0, block, n)] = rng.uniform(1.0, 50.0, n)
        y[np.arange(n), rng.integers(0, block, n)] = rng.uniform(1.0, 50.0, n)
    scale = 10.0 ** rng.uniform(-6, 3, (n, 1))            # tiny to large magnitudes (normalised y)
    return f32(y * scale)


@pytest.mark.parametrize("block", [16, 32, 64])
@pytest.mark.parametrize("wmse", [False, True])
@pytest.mark.parametrize("kind", ["laplace", "student_t", "normal", "repeated_max", "spiky"])
def test_loss_is_never_below_the_bound(block, wmse, kind):
    rng = np.random.default_rng(block * 7 + wmse * 3 + len(kind))
    n, segs = 400, block // 16
    y = blocks(kind, n, block, rng)
    w = f32(np.exp(rng.standard_normal((n, block))))
    if wmse:
        w[:, ::5] = 0.0                    # zero weights keep every term non-negative
    m = np.abs(y).max(-1)
    sbase = f32(m.astype(F64) / 6.0)
    vals = np.array([e4m3_value(c) for c in range(127)])
    I0 = np.clip(np.searchsorted(vals, sbase, side="right") - 1, 0, 126)
    lo = -3 if (not wmse and block == 16) else -8
    ys = y.reshape(n, segs, 16)
    ws = w.reshape(n, segs, 16)
    checked = 0
    for k in range(8 - lo):
        c = I0 + lo + k
        ok = (c >= 1) & (c <= 126)
        v = np.array([vals[ci] if 1 <= ci <= 126 else 1.0 for ci in c])
        L = group_sum(lane_loss(ys, ws, v[:, None, None], wmse), segs)
        bound = f32(group_sum(lane_bound(ys, ws, v[:, None], wmse), segs).astype(F64) * F64(MARGIN))
        assert np.all(L[ok] >= bound[ok]), (k, np.flatnonzero(ok & (L < bound))[:5])
        checked += int(ok.sum())
    assert checked > n


def test_a_double_counted_term_is_caught():
    """Planted mistake: counting the segment's largest element twice (both
    halves' terms taken from the overall maximum).  On blocks where one element
    carries nearly all of the loss the check above must then fail, so it is not
    vacuous."""
    rng = np.random.default_rng(5)
    n = 400
    y = blocks("spiky", n, 16, rng)
    w = f32(np.ones((n, 16)))
    m = np.abs(y).max(-1)
    vals = np.array([e4m3_value(c) for c in range(127)])
    I0 = np.clip(np.searchsorted(vals, f32(m.astype(F64) / 6.0), side="right") - 1, 0, 126)
    c = np.clip(I0 - 8, 1, 126)                       # saturating: the largest element dominates
    v = np.array([vals[ci] for ci in c])
    L = group_sum(lane_loss(y.reshape(n, 1, 16), w.reshape(n, 1, 16), v[:, None, None], False), 1)
    e = cand_err(m.astype(F32), v)
    wrong = f32(2.0 * f32(e.astype(F64) * e.astype(F64)).astype(F64) * F64(MARGIN))
    assert np.any(L < wrong)
