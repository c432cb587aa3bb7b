"""Pins for the LDLQ/GPTQ oracle (oracle/ldlq.py), all on the CPU.

What fixes the oracle, other than itself:
* its E2M1 rounding, E4M3 values, fixed-scale quantizer and dequantized values
  agree with the independent C oracle (nvfp4_oracle.c) element by element;
* the UDU^T factor reproduces the damped, reordered Hessian, and for n = 2 it is
  the closed form U_01 = b/c, D = (a - b^2/c, c);
* LDLQ and GPTQ's own form (inverse-Hessian Cholesky, in-place updates) give the
  same codes on correlated problems (QuIP's equivalence, Appendix A.2);
* a diagonal Hessian makes LDLQ plain rounding at the fixed scales;
* the proxy loss equals sum_k D_k |T_k - What_k|^2 (the LDL identity);
* the processing order is descending Hessian diagonal, ties by index;
* on correlated Hessians the error feedback lowers the proxy loss well below
  rounding at the same scales.
"""
import numpy as np
import pytest

import oracle
from oracle import ldlq as L


def rand_problem(m, n, seed, corr=0.9, ntok=None):
    rng = np.random.default_rng(seed)
    ntok = ntok or 4 * n
    # correlated, unevenly scaled input channels (AR(1) mixing, lognormal scales)
    Z = rng.standard_normal((ntok, n))
    X = np.empty_like(Z)
    X[:, 0] = Z[:, 0]
    for j in range(1, n):
        X[:, j] = corr * X[:, j - 1] + np.sqrt(1 - corr * corr) * Z[:, j]
    X *= np.exp(rng.standard_normal(n) * 0.7)[None, :]
    H = X.T @ X / ntok
    W = (rng.standard_normal((m, n)) * 0.02).astype(np.float32).astype(np.float64)
    return W, H


def fixed_scales(W, H, block=16):
    S, _ = oracle.global_scale(W.astype(np.float32), 256.0)
    w = np.diag(H).astype(np.float32)
    ref = oracle.quantize(oracle.METHOD_SCALESWEEP, W.astype(np.float32), block, S, oracle.WMSE, w=w)
    return S, ref["sf"]


def test_formats_match_c_oracle():
    for c in range(0, 127):
        assert L.e4m3_value(c) == oracle.e4m3_value(c)
    rng = np.random.default_rng(0)
    t = np.concatenate([rng.uniform(0, 8, 20000), [0.25, 0.75, 1.25, 1.75, 2.5, 3.5, 5.0, 6.0, 7.0, 1e30, 0.0]])
    t = t.astype(np.float32)
    got = L.rne_e2m1(t)
    ref = np.array([oracle.e2m1_rne(float(v)) for v in t])
    assert np.array_equal(got, ref & 7)


@pytest.mark.parametrize("seed", [1, 2])
def test_fixed_scale_quantizer_matches_c_oracle(seed):
    rng = np.random.default_rng(seed)
    rows, cols, block = 16, 128, 16
    x = (rng.standard_normal((rows, cols)) * 0.05).astype(np.float32)
    x[3, 5] = -0.0
    S, _ = oracle.global_scale(x, 256.0)
    ref = oracle.quantize(oracle.METHOD_SCALESWEEP, x, block, S)
    sf = ref["sf"].copy()
    sf[2, 1] = 0                                            # a zero-scale block: signed zeros
    sf[4, 3] = max(1, int(sf[4, 3]) - 9)                    # a scale far too small: saturation
    _, codes = oracle.block_losses_at(x, block, S, sf, want_codes=True)
    code_el = np.repeat(sf, block, axis=1)
    nib, val = L.quantize_fixed(x.astype(np.float64), S, code_el)
    packed = (nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8)
    assert np.array_equal(packed, codes)
    deq = oracle.dequantize(codes, sf, oracle.LAYOUT_LINEAR, S, rows, cols, block)
    assert np.array_equal(val.astype(np.float32).view(np.uint32), deq.view(np.uint32))


def test_udu_factor_and_two_by_two_closed_form():
    _, H = rand_problem(4, 48, 3)
    Hd, perm = L.damp_and_order(H)
    Hp = Hd[np.ix_(perm, perm)]
    U, D = L.udu(Hp)
    assert np.all(np.tril(U) == 0) and np.all(D > 0)
    I = np.eye(len(D))
    assert np.allclose((U + I) @ np.diag(D) @ (U + I).T, Hp, rtol=0, atol=1e-12 * np.abs(Hp).max())
    a, b, c = 3.0, -1.2, 2.0
    U2, D2 = L.udu(np.array([[a, b], [b, c]]))
    assert U2[0, 1] == pytest.approx(b / c, rel=1e-14)
    assert D2 == pytest.approx([a - b * b / c, c], rel=1e-14)


def test_two_column_feedback_closed_form():
    # w1's target is w1 + (w0 - What0) * b / c (the error of w0 pushed along H's coupling)
    H = np.array([[3.0, 1.1], [1.1, 2.0]])
    W = np.array([[0.37, -0.22], [1.05, 0.4], [-2.2, 2.9]])
    sf = np.full((3, 1), 56)                                  # one block, v = 1.0 (code 56)
    res = L.ldlq(W, H, 1.0, sf, block=2, alpha=0.0)
    assert list(res["perm"]) == [0, 1]
    w0q = L.quantize_fixed(W[:, 0], 1.0, np.full(3, 56), zero_positive=True)[1]
    t1 = W[:, 1] + (W[:, 0] - w0q) * (1.1 / 2.0)
    assert np.allclose(res["T"][:, 1], t1, rtol=1e-15)
    assert np.array_equal(res["What"][:, 1], L.quantize_fixed(t1, 1.0, np.full(3, 56), zero_positive=True)[1])


@pytest.mark.parametrize("seed", [4, 5, 6])
def test_ldlq_equals_gptq_form(seed):
    W, H = rand_problem(24, 96, seed)
    S, sf = fixed_scales(W, H)
    a = L.ldlq(W, H, S, sf)
    b = L.gptq(W, H, S, sf)
    assert np.array_equal(a["perm"], b["perm"])
    margin = L.decision_margin(a["T"], S, sf[:, a["perm"] // 16])
    differ = a["nib"][:, a["perm"]] != b["nib"][:, a["perm"]]
    assert not np.any(differ & (margin > 1e-9))
    assert differ.sum() == 0


def test_diagonal_hessian_is_rounding_at_fixed_scales():
    rng = np.random.default_rng(7)
    W = (rng.standard_normal((8, 64)) * 0.03).astype(np.float32)
    H = np.diag(np.exp(rng.standard_normal(64)))
    S, sf = fixed_scales(W.astype(np.float64), H)
    res = L.ldlq(W.astype(np.float64), H, S, sf)
    assert np.count_nonzero(res["U"]) == 0
    _, codes = oracle.block_losses_at(W, 16, S, sf, want_codes=True)
    nib = res["nib"]
    assert np.array_equal((nib[:, 0::2] | (nib[:, 1::2] << 4)).astype(np.uint8), codes)


@pytest.mark.parametrize("seed", [8, 9])
def test_proxy_loss_ldl_identity(seed):
    W, H = rand_problem(16, 80, seed)
    S, sf = fixed_scales(W, H)
    res = L.ldlq(W, H, S, sf)
    Hd, perm = L.damp_and_order(H)
    lhs = L.proxy_loss(W, res["What"], Hd)
    rhs = float(np.sum(res["D"][None, :] * (res["T"] - res["What"][:, perm]) ** 2))
    assert lhs == pytest.approx(rhs, rel=1e-10)
    # the targets are reproducible from the reconstructions alone
    assert np.allclose(L.targets(W, res["What"], perm, res["U"]), res["T"], rtol=0, atol=1e-13)


def test_static_order_descending_diagonal_stable():
    d = np.array([2.0, 5.0, 2.0, 7.0, 5.0, 1.0])
    _, perm = L.damp_and_order(np.diag(d))
    assert list(perm) == [3, 1, 4, 0, 2, 5]


def test_feedback_lowers_proxy_loss():
    W, H = rand_problem(64, 128, 11, corr=0.95)
    S, sf = fixed_scales(W, H)
    res = L.ldlq(W, H, S, sf)
    rtn = L.quantize_fixed(W, S, np.repeat(sf, 16, axis=1))[1]
    assert L.proxy_loss(W, res["What"], H) < 0.8 * L.proxy_loss(W, rtn, H)


def test_damping_is_one_percent_of_mean_diagonal():
    d = np.array([1.0, 2.0, 3.0, 10.0])
    Hd, _ = L.damp_and_order(np.diag(d))
    assert np.allclose(np.diag(Hd) - d, 0.01 * d.mean(), rtol=1e-15)


def test_planted_feedback_mistakes_are_caught(monkeypatch):
    """A flipped feedback sign or a transposed factor breaks the LDLQ = GPTQ pin."""
    W, H = rand_problem(16, 64, 12)
    S, sf = fixed_scales(W, H)
    ref = L.gptq(W, H, S, sf)["nib"]
    good = L.udu
    for bad in (lambda Hp: (-good(Hp)[0], good(Hp)[1]),
                lambda Hp: (np.triu(good(Hp)[0].T + good(Hp)[0], 1) * 0.5, good(Hp)[1]),
                lambda Hp: (good(Hp)[0] * 0.0, good(Hp)[1])):
        monkeypatch.setattr(L, "udu", bad)
        assert not np.array_equal(L.ldlq(W, H, S, sf)["nib"], ref)
    monkeypatch.setattr(L, "udu", good)
    assert np.array_equal(L.ldlq(W, H, S, sf)["nib"], ref)
