"""Helpers that compare the CUDA library's outputs with the CPU oracle.

Acceptance rule for codes and scales (bit-exact otherwise): where the oracle's
best and second-best window objectives differ by less than 1e-6 relative, the
GPU may pick another candidate if that candidate's oracle objective is within
1e-6 relative of the best; its nibbles must then equal the oracle's nibbles for
the GPU's scale.  Exact structural ties are resolved by the lowest code on both
sides and so are compared bit-exactly.
"""
import numpy as np
import torch

import oracle

REL = 1e-6


def to_np(t):
    if t is None:
        return None
    return t.detach().cpu().numpy()


def x_to_f32(x):
    return x.detach().cpu().float().numpy()


def compare_quantize(x, S, block, objective, w, w_row_stride, gpu, ref, method=0):
    """gpu: dict of torch tensors (codes, sf_linear[, sf_swizzled, block_loss]);
    ref: oracle.quantize(...) result on the same x and S.  Returns stats."""
    xs = x_to_f32(x) if isinstance(x, torch.Tensor) else x
    g_sf = to_np(gpu["sf_linear"]).reshape(-1)
    g_codes = to_np(gpu["codes"])
    r_sf = ref["sf"].reshape(-1)
    diff = np.nonzero(g_sf != r_sf)[0]
    stats = {"blocks": r_sf.size, "near_tie_accepted": int(diff.size)}
    wn = None if w is None else to_np(w)
    Lg = None
    if diff.size:
        best, second = ref["best"][diff], ref["second"][diff]
        gap_ok = (second - best) <= REL * np.abs(best)
        bad = diff[~gap_ok]
        assert bad.size == 0, (f"{bad.size} blocks differ beyond near-ties, e.g. block {bad[0]}: gpu {g_sf[bad[0]]} "
                               f"oracle {r_sf[bad[0]]} best {ref['best'][bad[0]]!r} second {ref['second'][bad[0]]!r}")
        # score the GPU's picks with the oracle, on the rows that hold them only
        rows, cols = xs.shape
        kb = cols // block
        rsel = np.unique(diff // kb)
        pos = np.searchsorted(rsel, diff // kb) * kb + diff % kb
        if wn is None or w_row_stride == 0:
            wsub = wn
        else:                                           # per-element weights: the selected rows' strides
            wf = wn.reshape(-1)
            wsub = np.zeros((rsel.size, w_row_stride), np.float32)
            for i, r in enumerate(rsel):
                seg = wf[r * w_row_stride:(r + 1) * w_row_stride]
                wsub[i, :seg.size] = seg
        Ls, cs = oracle.block_losses_at(xs[rsel], block, S, g_sf.reshape(rows, kb)[rsel], objective, w=wsub,
                                        w_row_stride=w_row_stride, want_codes=True)
        Lg = np.full(r_sf.size, np.nan)
        Lg[diff] = Ls[pos]
        assert np.all(Lg[diff] <= best * (1 + REL)), "GPU near-tie pick is not within 1e-6 of the best"
        # nibbles of differing blocks must match the oracle's nibbles for the GPU's scale
        cpb = block // 2
        gc = g_codes.reshape(-1, cpb)
        assert np.array_equal(gc[diff], cs.reshape(-1, cpb)[pos])
        same = np.ones(r_sf.size, bool)
        same[diff] = False
        assert np.array_equal(gc[same], ref["codes"].reshape(-1, cpb)[same])
    else:
        assert np.array_equal(g_codes, ref["codes"]), "codes differ although every scale matches"
    if gpu.get("sf_swizzled") is not None:
        assert np.array_equal(to_np(gpu["sf_swizzled"]), oracle.swizzle_scales(to_np(gpu["sf_linear"])))
    if gpu.get("block_loss") is not None:
        gl = to_np(gpu["block_loss"]).astype(np.float64)
        want = ref["best"].copy()
        if diff.size:
            want[diff] = Lg[diff]
        tol = 2e-6 * np.maximum(np.abs(want), 1e-30)
        assert np.all(np.abs(gl - want) <= tol + 1e-37), "per-block loss outside fp32 accumulation tolerance"
        tot_g, tot_r = gl.sum(), want.sum()
        assert abs(tot_g - tot_r) <= 1e-5 * abs(tot_r) + 1e-30
    return stats
