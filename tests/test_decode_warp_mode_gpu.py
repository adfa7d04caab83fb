"""Decode attention in the per-warp mode (batches of short (trajectory, KV head)
units: every consumer warp streams a slice of its own and ends its segments
alone), against the fp64 oracle on every row.

The planner takes the mode by itself; each test reads the planner's choice
from the workspace header (num_slices at byte 8, the mode flag at byte 56) to
make sure the mode it means to test is the one that ran.  Cases: short units
only; short units with a few long trajectories that span several warp slices
(their partials go through the last-arrival merge); a batch just above the
mode's minimum size, with a handful of page-heads per warp; head_dim 64 with a
group of 8; repeat calls bit-identical; a plan serving several runs; the fused
append.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300.workloads import bf16_bits
from _gpu_util import abs_bits, assert_close_bounded, device_tensors, make_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def _header(ws):
    h = ws[:64].cpu().numpy()
    return int(h[8:12].view(np.int32)[0]), int(h[56:60].view(np.int32)[0])


def _run(batch, tensors=None):
    q, k, v, bt, cl = tensors if tensors is not None else device_tensors(batch)
    ws = torch.empty(cadkv.decode_attention_workspace_size(q.shape[0], q.shape[1], k.shape[1],
                                                           q.shape[2], bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    out, lse = cadkv.decode_attention(q, k, v, bt, cl, workspace=ws)
    torch.cuda.synchronize()
    assert cadkv.decode_attention_status(ws) == 0
    return out, lse, ws


def _check(batch, out, lse, what):
    qb, kb, vb = bf16_bits(batch.q), bf16_bits(batch.k_pages), bf16_bits(batch.v_pages)
    ref, ref_lse = oracle.decode_attention(qb, kb, vb, batch.block_table, batch.context_lens)
    absv, _ = oracle.decode_attention(qb, kb, abs_bits(vb), batch.block_table,
                                      batch.context_lens)
    assert_close_bounded(out, lse, ref, ref_lse, absv, what)


def _warp_slices():
    return cadkv.library().cadkv_device_sms() * 8


@pytest.mark.parametrize("hq,hkv,d,seed", [(32, 8, 128, 600), (40, 8, 128, 601),
                                          (16, 2, 64, 602)])
def test_short_units_every_row(hq, hkv, d, seed):
    rng = np.random.Generator(np.random.PCG64(seed))
    lens = rng.integers(0, 401, 2500).astype(np.int32)
    batch = make_batch(lens, hq, hkv, d, seed=seed + 10)
    out, lse, ws = _run(batch)
    slices, mode = _header(ws)
    assert mode == 1 and slices == _warp_slices()
    _check(batch, out, lse, f"per-warp mode, {hq}/{hkv} heads, D={d}")


def test_short_units_with_long_trajectories_every_row():
    """Four 9,000-token trajectories among 3,000 short ones: each of their units
    spans several warp slices, so their partials are merged by the warp that
    delivers the last one."""
    rng = np.random.Generator(np.random.PCG64(610))
    lens = rng.integers(1, 65, 3000).astype(np.int32)
    lens[[5, 700, 1999, 2999]] = 9000
    batch = make_batch(lens, 32, 8, 128, seed=611)
    out, lse, ws = _run(batch)
    slices, mode = _header(ws)
    assert mode == 1 and slices == _warp_slices()
    W = int((-(-lens.astype(np.int64) // 16)).sum()) * 8
    assert 9000 // 16 > 2 * W // slices        # a long unit spans more than two slices
    _check(batch, out, lse, "per-warp mode with long trajectories")


def test_few_page_heads_per_warp_every_row():
    """A batch just large enough for the mode: 90 trajectories of 100-250
    tokens give each warp slice a handful of page-heads, so nearly every unit is
    cut across two or three warps and merged by the last one."""
    rng = np.random.Generator(np.random.PCG64(615))
    lens = rng.integers(100, 251, 90).astype(np.int32)
    batch = make_batch(lens, 32, 8, 128, seed=616)
    out, lse, ws = _run(batch)
    slices, mode = _header(ws)
    assert mode == 1 and slices == _warp_slices()
    W = int((-(-lens.astype(np.int64) // 16)).sum()) * 8
    assert W < 8 * slices                      # fewer than 8 page-heads per warp slice
    _check(batch, out, lse, "per-warp mode, few page-heads per warp")


def test_group_of_eight_head_dim_64():
    rng = np.random.Generator(np.random.PCG64(620))
    lens = rng.integers(1, 200, 4000).astype(np.int32)
    batch = make_batch(lens, 16, 2, 64, seed=621)
    out, lse, ws = _run(batch)
    assert _header(ws)[1] == 1
    _check(batch, out, lse, "per-warp mode, G=8, D=64")


def test_repeat_calls_and_plan_runs_are_bit_identical():
    """Static warp slices: the same bits call after call, and one plan serving
    several runs gives the single call's bits."""
    rng = np.random.Generator(np.random.PCG64(630))
    lens = rng.integers(1, 300, 2000).astype(np.int32)
    lens[17] = 5000
    batch = make_batch(lens, 32, 8, 128, seed=631)
    tensors = device_tensors(batch)
    out_a, lse_a, ws = _run(batch, tensors)
    assert _header(ws)[1] == 1
    out_b, lse_b, _ = _run(batch, tensors)
    assert torch.equal(out_a, out_b) and torch.equal(lse_a, lse_b)
    q, k, v, bt, cl = tensors
    out_c, lse_c = torch.empty_like(out_a), torch.empty_like(lse_a)
    cadkv.decode_attention_plan(q, k, v, bt, cl, out_c, lse_c, ws)
    for _ in range(3):
        out_c.fill_(float("nan"))
        cadkv.decode_attention_run(q, k, v, bt, cl, out_c, lse_c, ws)
        torch.cuda.synchronize()
        assert torch.equal(out_a, out_c) and torch.equal(lse_a, lse_c)
    assert cadkv.decode_attention_status(ws) == 0


def test_append_in_per_warp_mode():
    """The fused append followed by the per-warp attention: pool bit-exact
    against the oracle's append, attention against the oracle on every row."""
    rng = np.random.Generator(np.random.PCG64(640))
    lens = rng.integers(1, 200, 3000).astype(np.int32)
    batch = make_batch(lens, 32, 8, 128, seed=641)
    g = torch.Generator().manual_seed(642)
    k_new = torch.randn((3000, 8, 128), generator=g).to(torch.bfloat16)
    v_new = torch.randn((3000, 8, 128), generator=g).to(torch.bfloat16)
    kp = bf16_bits(batch.k_pages).copy()
    vp = bf16_bits(batch.v_pages).copy()
    oracle.kv_append(kp, vp, bf16_bits(k_new), bf16_bits(v_new), batch.block_table,
                     batch.context_lens)
    k_dev, v_dev = batch.k_pages.cuda(), batch.v_pages.cuda()
    out, lse = cadkv.decode_attention_append(
        batch.q.cuda(), k_new.cuda(), v_new.cuda(), k_dev, v_dev,
        torch.from_numpy(batch.block_table).cuda(), torch.from_numpy(batch.context_lens).cuda())
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bf16_bits(k_dev), kp)
    np.testing.assert_array_equal(bf16_bits(v_dev), vp)
    qb = bf16_bits(batch.q)
    ref, ref_lse = oracle.decode_attention(qb, kp, vp, batch.block_table, batch.context_lens)
    absv, _ = oracle.decode_attention(qb, kp, abs_bits(vp), batch.block_table,
                                      batch.context_lens)
    assert_close_bounded(out, lse, ref, ref_lse, absv, "append, per-warp mode")
