"""GPU decode step with the fused KV append (decode_attention_append) against
the oracle: the pool after the append is bit-identical to the oracle's
kv_append, and the attention over it is within the parity tolerances."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS
from paper_2609_36899_gb300.workloads import MIXED, bf16_bits, make_decode_batch
from _gpu_util import assert_close, full_oracle, make_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def _new_rows(batch, hkv, d, seed):
    g = torch.Generator().manual_seed(seed)
    k = torch.randn((batch, hkv, d), generator=g).to(torch.bfloat16)
    v = torch.randn((batch, hkv, d), generator=g).to(torch.bfloat16)
    return k, v


@pytest.mark.parametrize("g,d", [(1, 64), (4, 128), (8, 128), (8, 64)])
def test_append_then_attend(g, d):
    lens = [0, 1, 2, 16, 17, 100, 4096, 31]
    hkv = 2
    batch = make_batch(lens, g * hkv, hkv, d, seed=300 + g + d)   # NaN in the new slots
    k_new, v_new = _new_rows(len(lens), hkv, d, seed=301 + g + d)
    kp = bf16_bits(batch.k_pages).copy()
    vp = bf16_bits(batch.v_pages).copy()
    oracle.kv_append(kp, vp, bf16_bits(k_new), bf16_bits(v_new), batch.block_table,
                     batch.context_lens)
    q = batch.q.cuda()
    k_dev, v_dev = batch.k_pages.cuda(), batch.v_pages.cuda()
    bt = torch.from_numpy(batch.block_table).cuda()
    cl = torch.from_numpy(batch.context_lens).cuda()
    out, lse = cadkv.decode_attention_append(q, k_new.cuda(), v_new.cuda(), k_dev, v_dev, bt, cl)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bf16_bits(k_dev), kp)
    np.testing.assert_array_equal(bf16_bits(v_dev), vp)
    ref, ref_lse = oracle.decode_attention(bf16_bits(batch.q), kp, vp, batch.block_table,
                                           batch.context_lens)
    assert_close(out, lse, ref, ref_lse, f"append G={g} D={d}")


def test_append_large_batch():
    """3,000 trajectories x 4 KV heads: 375 append CTAs beside the 1,024-thread
    planner.  The pool after the append equals the oracle's kv_append, and the
    attention over it matches the oracle on every row."""
    rng = np.random.Generator(np.random.PCG64(330))
    lens = rng.integers(0, 300, 3000).astype(np.int32)
    batch = make_batch(lens, 16, 4, 64, seed=331)
    k_new, v_new = _new_rows(3000, 4, 64, seed=332)
    kp = bf16_bits(batch.k_pages).copy()
    vp = bf16_bits(batch.v_pages).copy()
    oracle.kv_append(kp, vp, bf16_bits(k_new), bf16_bits(v_new), batch.block_table,
                     batch.context_lens)
    q = batch.q.cuda()
    k_dev, v_dev = batch.k_pages.cuda(), batch.v_pages.cuda()
    bt = torch.from_numpy(batch.block_table).cuda()
    cl = torch.from_numpy(batch.context_lens).cuda()
    out, lse = cadkv.decode_attention_append(q, k_new.cuda(), v_new.cuda(), k_dev, v_dev, bt, cl)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bf16_bits(k_dev), kp)
    np.testing.assert_array_equal(bf16_bits(v_dev), vp)
    ref, ref_lse = oracle.decode_attention(bf16_bits(batch.q), kp, vp, batch.block_table,
                                           batch.context_lens)
    assert_close(out, lse, ref, ref_lse, "append, B = 3000")


def test_append_full_size_mixed_every_row():
    """The whole decode step of the full-size mixed batch (512 trajectories,
    dynamic-slice path).  The pool after the append equals the oracle's
    kv_append of the original pool (every trajectory's last page compared bit
    for bit with the oracle applied to a host copy of it; every other page
    unchanged), and every output row is within tolerance of the oracle's
    attention over that pool."""
    batch = make_decode_batch(MIXED, device="cuda")
    g = torch.Generator(device="cuda").manual_seed(4242)
    k_new = torch.randn((MIXED.batch, 8, 128), generator=g, device="cuda").to(torch.bfloat16)
    v_new = torch.randn((MIXED.batch, 8, 128), generator=g, device="cuda").to(torch.bfloat16)
    lens = batch.context_lens
    last = np.array([batch.block_table[b, (int(n) - 1) // 16] for b, n in enumerate(lens)],
                    dtype=np.int64)
    assert len(set(last.tolist())) == len(last)      # one distinct page per trajectory
    last_dev = torch.from_numpy(last).cuda()
    k_before = batch.k_pages.clone()
    v_before = batch.v_pages.clone()
    bt = torch.from_numpy(batch.block_table).cuda()
    cl = torch.from_numpy(lens).cuda()
    out, lse = cadkv.decode_attention_append(batch.q, k_new, v_new, batch.k_pages,
                                             batch.v_pages, bt, cl)
    torch.cuda.synchronize()
    # oracle append on host copies of the last pages, renumbered 0..B-1 (every
    # page of row b names copy b; only the last one is written)
    table = np.full_like(batch.block_table, -1)
    for b, n in enumerate(lens):
        table[b, :-(-int(n) // 16)] = b
    kp = bf16_bits(k_before.index_select(0, last_dev)).copy()
    vp = bf16_bits(v_before.index_select(0, last_dev)).copy()
    oracle.kv_append(kp, vp, bf16_bits(k_new), bf16_bits(v_new), table, lens)
    np.testing.assert_array_equal(bf16_bits(batch.k_pages.index_select(0, last_dev)), kp)
    np.testing.assert_array_equal(bf16_bits(batch.v_pages.index_select(0, last_dev)), vp)
    for after, before in ((batch.k_pages, k_before), (batch.v_pages, v_before)):
        changed = (after.view(torch.int16) != before.view(torch.int16)).flatten(1).any(1)
        assert set(changed.nonzero().flatten().tolist()) <= set(last.tolist())
    del k_before, v_before
    ref, ref_lse = full_oracle(batch)               # over the verified pool
    assert_close(out, lse, ref, ref_lse, "mixed + append, all rows")
    del batch
    torch.cuda.empty_cache()


def test_append_bad_last_page_is_reported_and_not_written():
    batch = make_batch([20, 40], 4, 1, 64, seed=310, nan_tails=False)
    k_new, v_new = _new_rows(2, 1, 64, seed=311)
    q = batch.q.cuda()
    k_dev, v_dev = batch.k_pages.cuda(), batch.v_pages.cuda()
    bt = torch.from_numpy(batch.block_table).cuda()
    cl = torch.from_numpy(batch.context_lens).cuda()
    bt[1, 2] = batch.num_pages + 3               # last page of trajectory 1
    k_before = k_dev.clone()
    ws = torch.empty(cadkv.decode_attention_workspace_size(2, 4, 1, 64, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    cadkv.decode_attention_append(q, k_new.cuda(), v_new.cuda(), k_dev, v_dev, bt, cl,
                                  workspace=ws)
    assert cadkv.decode_attention_status(ws) == STATUS["CADKV_ERR_OOB"]
    # only trajectory 0's new slot changed
    t0 = 19
    ph0 = int(batch.block_table[0, t0 // 16])
    changed = (k_dev.view(torch.int16) != k_before.view(torch.int16))
    assert changed.any(dim=-1).nonzero().tolist() == [[ph0, 0, t0 % 16]]
