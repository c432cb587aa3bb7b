"""The multi-GPU row partition (nvfp4_row_shard_layout, paper_2606_07618_gb300/shard.py)
on CPU: no kernel runs here, the oracle stands in for the GPU's quantisation.

* The layout: shards cover the rows exactly once, boundaries fall on multiples
  of 128 rows, and the output offsets tile the whole tensor's codes, linear
  scales and swizzled-scale atoms.
* Blocks are independent given S (Sec. 4.2.1): every shard quantised alone with
  the whole tensor's S, placed at its offsets, reproduces the whole tensor's
  oracle result byte for byte, swizzled atoms included.
* With two gloo ranks, shard.allreduce_scale (the collective the GPU path uses)
  turns the shards' own global scales and status words into the whole tensor's
  S bit for bit and the OR of the flags, and the ranks' shards, gathered, equal
  the single-tensor result.
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def B():
    from paper_2606_07618_gb300 import binding
    binding.lib()
    return binding


@pytest.mark.parametrize("rows,cols,block", [(1000, 256, 16), (128, 64, 16), (300, 192, 32), (2049, 512, 64),
                                             (5, 64, 16), (0, 64, 16)])
@pytest.mark.parametrize("world", [1, 2, 3, 8, 40])
def test_row_shard_layout_tiles_the_tensor(B, rows, cols, block, world):
    kb = cols // block
    kpad4 = (kb + 3) // 4
    sw_total = ((rows + 127) // 128) * kpad4 * 512
    covered, prev_end, sw_next = 0, 0, 0
    for rank in range(world):
        lay = B.nvfp4_row_shard_layout(rows, cols, block, world, rank)
        assert lay.row_begin == prev_end and lay.row_end >= lay.row_begin
        assert lay.row_begin % 128 == 0 or lay.row_begin == rows
        assert lay.row_end % 128 == 0 or lay.row_end == rows
        assert lay.x_offset == lay.row_begin * cols
        assert lay.codes_offset == lay.row_begin * cols // 2
        assert lay.sf_linear_offset == lay.row_begin * kb
        if block == 16:
            assert lay.sf_swizzled_offset == sw_next
            sw_next += lay.sf_swizzled_bytes
        else:
            assert lay.sf_swizzled_offset == -1 and lay.sf_swizzled_bytes == -1
        covered += lay.row_end - lay.row_begin
        prev_end = lay.row_end
    assert covered == rows and prev_end == rows
    if block == 16:
        assert sw_next == sw_total
    # balanced: shards differ by at most one 128-row block
    sizes = [B.nvfp4_row_shard_layout(rows, cols, block, world, r) for r in range(world)]
    blocks = [(s.row_end - s.row_begin + 127) // 128 for s in sizes]
    assert max(blocks) - min(blocks) <= 1


def test_row_shard_layout_rejects_bad_arguments(B):
    from paper_2606_07618_gb300.binding import Nvfp4Error
    for args in ((100, 64, 16, 0, 0), (100, 64, 16, 2, 2), (100, 64, 16, 2, -1), (100, 40, 16, 2, 0),
                 (100, 64, 8, 2, 0), (-1, 64, 16, 2, 0)):
        with pytest.raises(Nvfp4Error):
            B.nvfp4_row_shard_layout(*args)


def _shard_outputs_by_oracle(x, S, block, objective, w, world):
    """Quantise each shard alone (oracle, whole-tensor S) and place its outputs
    at the layout's offsets in full-size buffers."""
    import oracle
    from paper_2606_07618_gb300 import binding as B
    rows, cols = x.shape
    kb = cols // block
    codes = np.full((rows, cols // 2), 0xEE, np.uint8)
    sf = np.full((rows, kb), 0xEE, np.uint8)
    sw = np.full(oracle.swizzle_bytes(rows, kb), 0xEE, np.uint8) if block == 16 else None
    for rank in range(world):
        lay = B.nvfp4_row_shard_layout(rows, cols, block, world, rank)
        r0, r1 = lay.row_begin, lay.row_end
        if r1 == r0:
            continue
        o = oracle.quantize(0, x[r0:r1], block, S, objective, w=w)
        codes[r0:r1] = o["codes"]
        sf[r0:r1] = o["sf"]
        if sw is not None:
            part = oracle.swizzle_scales(o["sf"])
            assert part.size == lay.sf_swizzled_bytes
            sw[lay.sf_swizzled_offset:lay.sf_swizzled_offset + part.size] = part
    return codes, sf, sw


@pytest.mark.parametrize("world", [2, 3, 5])
@pytest.mark.parametrize("block,objective", [(16, 0), (16, 1), (32, 1), (64, 0)])
def test_shards_reassemble_the_whole_tensor(B, world, block, objective):
    import oracle
    from paper_2606_07618_gb300 import workloads as W
    x = W.small_tensor(650, 256, 77, dist="laplace", std=0.015, outliers=2, mult=30.0).float().numpy()
    w = np.exp(np.random.default_rng(4).standard_normal(256)).astype(np.float32) if objective else None
    S, _ = oracle.global_scale(x, 256.0)
    whole = oracle.quantize(0, x, block, S, objective, w=w)
    codes, sf, sw = _shard_outputs_by_oracle(x, S, block, objective, w, world)
    assert np.array_equal(codes, whole["codes"]) and np.array_equal(sf, whole["sf"])
    if sw is not None:
        assert np.array_equal(sw, oracle.swizzle_scales(whole["sf"]))


# --------------------------------------------------------------------------- two gloo ranks
def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_worker(rank, world, port, q, plant_nan):
    """One rank: its shard's own S and status (oracle), the library's
    collective, then its shard's quantisation with the reduced S."""
    sys.path.insert(0, ROOT)
    sys.path.insert(0, os.path.join(ROOT, "tests"))
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from paper_2606_07618_gb300 import shard
    from paper_2606_07618_gb300 import workloads as W
    x = W.small_tensor(900, 192, 55, dist="student_t", std=1.0, outliers=3, mult=40.0).float().numpy()
    if plant_nan:
        x[700, 5] = np.nan                               # in the last shard only
    lay = shard.layout(x.shape[0], x.shape[1], 16, world, rank)
    xs = x[lay.row_begin:lay.row_end]
    S_k, bad = oracle.global_scale(xs, 256.0) if xs.size else (0.0, False)
    buf = torch.tensor([np.float32(S_k).view(np.int32), int(bad)], dtype=torch.int32)
    shard.allreduce_scale(buf)
    S = float(shard.global_scale_of(buf).item())
    o = oracle.quantize(0, xs, 16, S, oracle.MSE) if xs.size else None
    q.put((rank, lay.row_begin, lay.row_end, S, int(buf[1].item()), None if o is None else o["codes"],
           None if o is None else o["sf"]))
    dist.barrier()
    dist.destroy_process_group()


@pytest.mark.parametrize("plant_nan", [False, True])
def test_two_gloo_ranks_reduce_the_scale_and_reassemble(plant_nan):
    import oracle
    from paper_2606_07618_gb300 import workloads as W
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_worker, args=(r, world, port, q, plant_nan)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=180) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    x = W.small_tensor(900, 192, 55, dist="student_t", std=1.0, outliers=3, mult=40.0).float().numpy()
    if plant_nan:
        x[700, 5] = np.nan
    S, bad = oracle.global_scale(x, 256.0)
    whole = oracle.quantize(0, x, 16, S, oracle.MSE)
    assert [r[3] for r in res] == [np.float32(S)] * world          # every rank holds the whole tensor's S
    assert [r[4] for r in res] == [int(bad)] * world                # and the OR of the status words
    assert res[0][1] == 0 and res[0][2] == res[1][1] == 512 and res[1][2] == 900
    codes = np.concatenate([r[5] for r in res])
    sf = np.concatenate([r[6] for r in res])
    assert np.array_equal(codes, whole["codes"]) and np.array_equal(sf, whole["sf"])
