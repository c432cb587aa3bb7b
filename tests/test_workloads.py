"""The seeded synthetic workloads match their stated recipe (CPU).

Shapes of every configuration; the outlier-column counts round(frac * in);
determinism and row-slice consistency of the draws; and the value
distributions, checked by moments on samples: N(0, 0.02^2), Student-t(3)
(heavy tails: no finite fourth moment), Laplace(0, b) (E|x| = b), the per-head
factor of the K/V/Q tensors, and lognormal(0, 1) channel weights.
"""
import math

import numpy as np
import pytest
import torch

from paper_2606_07618_gb300 import workloads as W


def test_shapes_of_every_configuration():
    shapes = {wl: [(t.rows, t.cols) for t in W.workload(wl).tensors] for wl in W.ALL_CONFIGS}
    assert shapes["weight-2048"] == [(2048, 2048)]
    assert shapes["llama8b"] == [(4096, 4096), (1024, 4096), (1024, 4096), (4096, 4096), (14336, 4096),
                                 (14336, 4096), (4096, 14336)]
    assert W.workload("llama8b").numel == 218103808
    assert shapes["act-8192"] == [(8192, 4096)]
    assert shapes["kvq"] == [(16 * 8 * 4096, 128), (16 * 8 * 4096, 128), (16 * 32 * 4096, 128)]
    for b in (16, 32, 64):
        for o in ("mse", "wmse"):
            wl = W.workload(f"qwen72b-b{b}-{o}")
            assert [(t.rows, t.cols) for t in wl.tensors] == [(8192, 29568), (29568, 8192)]
            assert wl.block == b and wl.objective == o
    assert W.workload("weight-2048").fp8_div == 448.0
    assert all(W.workload(wl).fp8_div == 256.0 for wl in W.ALL_CONFIGS if wl != "weight-2048")
    assert W.workload("llama8b").objective == "wmse" and W.workload("act-8192").dynamic_scale


def test_outlier_column_counts():
    ts = {t.name: t for t in W.workload("llama8b").tensors}
    g = torch.Generator().manual_seed(0)
    assert W._outlier_cols(ts["q"], g).numel() == 4          # round(0.001 * 4096)
    assert W._outlier_cols(ts["down"], g).numel() == 14      # round(0.001 * 14336)
    q = {t.name: t for t in W.workload("qwen72b-b16-mse").tensors}
    assert W._outlier_cols(q["w_8192x29568"], g).numel() == 15   # round(0.0005 * 29568)
    assert W._outlier_cols(q["w_29568x8192"], g).numel() == 4    # round(0.0005 * 8192)
    assert W._outlier_cols(W.workload("act-8192").tensors[0], g).numel() == 16


def test_draws_are_deterministic_and_row_slices_agree():
    t = W.Tensor("t", 300, 256, "laplace", 77, std=0.015, outlier_frac=0.01, outlier_mult=30.0)
    a, b = W.draw(t), W.draw(t)
    assert a.dtype == torch.bfloat16 and a.shape == (300, 256)
    assert torch.equal(a, b)
    assert torch.equal(W.draw(t, rows=slice(0, 100)), a[:100])
    t2 = W.Tensor("t", 300, 256, "laplace", 78, std=0.015)
    assert not torch.equal(W.draw(t2), a)


def test_normal_recipe_and_outlier_columns():
    t = W.Tensor("t", 2048, 1024, "normal", 5, std=0.02, outlier_frac=0.004, outlier_mult=20.0)
    x = W.draw(t).float().numpy()
    col_std = x.std(axis=0)
    big = col_std > 0.1
    assert big.sum() == 4                                     # round(0.004 * 1024) columns x20
    assert col_std[big] == pytest.approx(np.full(4, 0.4), rel=0.1)
    assert x[:, ~big].std() == pytest.approx(0.02, rel=0.01)
    assert abs(x[:, ~big].mean()) < 0.001


def test_student_t_recipe_is_heavy_tailed():
    t = W.Tensor("t", 4096, 512, "student_t", 9)
    x = W.draw(t).float().numpy().ravel()
    # t(3): variance 3, P(|x| > 5) = 0.0154 (from the t(3) CDF); a normal would give ~6e-7
    assert x.var() == pytest.approx(3.0, rel=0.25)
    assert np.mean(np.abs(x) > 5.0) == pytest.approx(0.0154, rel=0.1)
    assert np.median(np.abs(x)) == pytest.approx(0.7649, rel=0.03)      # t(3) quartile


def test_laplace_recipe():
    t = W.Tensor("t", 4096, 512, "laplace", 11, std=0.015)
    x = W.draw(t).float().numpy().ravel()
    assert np.mean(np.abs(x)) == pytest.approx(0.015, rel=0.01)         # E|x| = b
    assert np.median(np.abs(x)) == pytest.approx(0.015 * math.log(2), rel=0.02)
    assert abs(np.mean(x)) < 2e-4 and np.isfinite(x).all()


def test_kvq_per_head_factor():
    t = W.workload("kvq").tensors[0]
    rows = slice(0, 8 * 4096)                                 # first batch: 8 heads x 4096 positions
    x = W.draw(t, rows=rows).float().numpy()
    head_std = x.reshape(8, 4096 * 128).std(axis=1)
    g = W._gen(t.seed)
    want = torch.exp(0.5 * torch.randn(8, generator=g)).numpy()
    assert head_std == pytest.approx(want, rel=0.02)


def test_lognormal_channel_weights():
    t = W.Tensor("t", 4, 200000, "normal", 3, weights=True)
    w = W.draw_weights(t).numpy()
    lw = np.log(w)
    assert lw.mean() == pytest.approx(0.0, abs=0.01) and lw.std() == pytest.approx(1.0, rel=0.01)
