"""GPU chunked prefill attention (tcgen05 kernel, through the C ABI) against
the fp64 oracle on the same bf16 inputs, within the decode tolerances."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS
from paper_2609_36899_gb300.workloads import bf16_bits
from _gpu_util import assert_close, make_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def _case(lens, chunks, hq, hkv, seed):
    batch = make_batch(lens, hq, hkv, 128, seed=seed)     # NaN past n_b in the pool
    offs = np.concatenate([[0], np.cumsum(chunks)]).astype(np.int64)
    g = torch.Generator().manual_seed(seed + 1)
    q = torch.randn((int(offs[-1]), hq, 128), generator=g).to(torch.bfloat16)
    return batch, offs, q


def _run(batch, offs, q):
    out, lse, ws = cadkv.prefill_attention(
        q.cuda(), torch.from_numpy(offs).cuda(), batch.k_pages.cuda(), batch.v_pages.cuda(),
        torch.from_numpy(batch.block_table).cuda(), torch.from_numpy(batch.context_lens).cuda())
    torch.cuda.synchronize()
    return out, lse, ws


def _oracle(batch, offs, q):
    return oracle.prefill_attention(bf16_bits(q), offs, bf16_bits(batch.k_pages),
                                    bf16_bits(batch.v_pages), batch.block_table,
                                    batch.context_lens)


@pytest.mark.parametrize("g", [1, 2, 3, 4, 5, 6, 7, 8])
def test_prefill_small(g):
    lens, chunks = [40, 300, 17, 130], [40, 5, 17, 129]
    batch, offs, q = _case(lens, chunks, 2 * g, 2, seed=400 + g)
    out, lse, ws = _run(batch, offs, q)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, f"prefill G={g}")


def test_prefill_many_tiles():
    """Chunks spanning several query tiles and key tiles, ragged everywhere."""
    lens, chunks = [1000, 700, 257], [300, 1, 257]
    batch, offs, q = _case(lens, chunks, 8, 2, seed=410)
    out, lse, ws = _run(batch, offs, q)
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill many tiles")


def test_prefill_many_trajectories():
    """1,500 trajectories (the 1,024-thread planner scans their work items in two
    rounds), contexts U[1, 400], chunks of 1..24 tokens: many small items, with
    the last partial wave split; every row against the oracle."""
    rng = np.random.Generator(np.random.PCG64(430))
    lens = rng.integers(1, 401, 1500)
    chunks = np.minimum(lens, rng.integers(1, 25, 1500))
    batch, offs, q = _case(lens.tolist(), chunks.tolist(), 8, 2, seed=431)
    out, lse, ws = _run(batch, offs, q)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill, 1,500 trajectories")


def test_prefill_qwen_shape():
    """32 query / 8 KV heads (G = 4), contexts of a few thousand tokens."""
    lens, chunks = [3000, 4500], [256, 130]
    batch, offs, q = _case(lens, chunks, 32, 8, seed=420)
    out, lse, ws = _run(batch, offs, q)
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill 32/8")


def test_prefill_qwen14b_shape():
    """40 query / 8 KV heads (G = 5: a tile holds 25 tokens, 125 rows + 3 padding
    rows), chunks spanning several query tiles and items, ragged tails."""
    lens, chunks = [3000, 1200, 60], [200, 77, 60]
    batch, offs, q = _case(lens, chunks, 40, 8, seed=425)
    out, lse, ws = _run(batch, offs, q)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill 40/8")


def test_prefill_full_size_every_row():
    """The bench's prefill workload (8 trajectories x last 512 of 16,384 tokens,
    32/8 heads, D = 128) in the bench's launch configuration: every query token
    of every trajectory, every head, against the oracle."""
    from paper_2609_36899_gb300.workloads import PREFILL, make_prefill_job
    w = PREFILL
    b, offs, q = make_prefill_job(w, "cuda")
    bt = torch.from_numpy(b.block_table).cuda()
    cl = torch.from_numpy(b.context_lens).cuda()
    out, lse, ws = cadkv.prefill_attention(q, offs, b.k_pages, b.v_pages, bt, cl)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = oracle.prefill_attention(bf16_bits(q), offs.cpu().numpy(),
                                            bf16_bits(b.k_pages), bf16_bits(b.v_pages),
                                            b.block_table, b.context_lens)
    assert ref.shape == tuple(out.shape)
    assert_close(out, lse, ref, ref_lse, "prefill workload, all rows")
    del b, q, out
    torch.cuda.empty_cache()


@pytest.mark.parametrize("direction", [1.0, -1.0])
def test_prefill_running_max_moves(direction):
    """Scores that rise (or fall) steadily along the context.  Rising: every key
    tile lifts each row's max by ~16 log2 units, so P taken against the previous
    max is far too large and must be recomputed against the new one.  Falling:
    the first key tile holds the max throughout."""
    lens, chunks = [1500, 700], [300, 129]
    batch, offs, q = _case(lens, chunks, 2, 2, seed=460)
    q.fill_(0.25)
    kp = batch.k_pages.float()
    for b, n in enumerate(lens):
        npg = (n + 15) // 16
        pages = torch.from_numpy(batch.block_table[b, :npg].astype(np.int64))
        c = direction * torch.arange(n, dtype=torch.float32) / 16.0
        for h in range(2):
            blk = kp[pages, h].reshape(npg * 16, 128)    # a copy; slots past n stay NaN
            blk[:n] = 0.5 * c[:, None] + 0.05 * blk[:n]  # aligned with q, plus noise
            kp[pages, h] = blk.reshape(npg, 16, 128)
    batch.k_pages = kp.to(torch.bfloat16)
    out, lse, ws = _run(batch, offs, q)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, f"prefill, running max direction {direction}")


def test_prefill_items_split_many_ways():
    """Fewer work items than SMs, each with many key tiles: every item is cut into
    the most pieces (16 here, 40,960 keys = 320 tiles per item), each piece stores
    its partial rows and the last one to finish merges all of them."""
    lens, chunks = [40960], [64]
    batch, offs, q = _case(lens, chunks, 8, 1, seed=470)   # G = 8: 2 items of 32 tokens
    out, lse, ws = _run(batch, offs, q)
    assert cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill split 16 ways")


def test_prefill_chunk_of_one_matches_decode():
    lens = [77, 1, 513]
    batch, offs, q = _case(lens, [1, 1, 1], 16, 2, seed=430)
    out, lse, _ = _run(batch, offs, q)
    dq = q.view(3, 16, 128).cuda()
    dec_out, dec_lse = cadkv.decode_attention(
        dq, batch.k_pages.cuda(), batch.v_pages.cuda(),
        torch.from_numpy(batch.block_table).cuda(), torch.from_numpy(batch.context_lens).cuda())
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, lse, ref, ref_lse, "prefill C=1")
    assert_close(dec_out, dec_lse, ref.reshape(3, 16, 128), ref_lse.reshape(3, 16), "decode")


def test_prefill_rejects_chunk_longer_than_context():
    batch, offs, q = _case([20, 40], [5, 10], 4, 1, seed=440)
    cl = torch.from_numpy(batch.context_lens).cuda()
    cl[1] = 7                      # chunk of 10 cannot end at position 6
    out = torch.full((15, 4, 128), 3.0, dtype=torch.bfloat16, device="cuda")
    _, _, ws = cadkv.prefill_attention(
        q.cuda(), torch.from_numpy(offs).cuda(), batch.k_pages.cuda(), batch.v_pages.cuda(),
        torch.from_numpy(batch.block_table).cuda(), cl, out=out)
    assert cadkv.prefill_attention_status(ws) == STATUS["CADKV_ERR_SHAPE"]
    assert torch.all(out[5:] == 3.0)                     # trajectory 1 untouched
    ref, ref_lse = oracle.prefill_attention(
        bf16_bits(q[:5]), offs[:2], bf16_bits(batch.k_pages), bf16_bits(batch.v_pages),
        batch.block_table[:1], batch.context_lens[:1])
    assert_close(out[:5], None, ref, ref_lse, "trajectory 0")


def test_prefill_zero_length_chunks_and_no_lse():
    """Trajectories that re-prefill nothing sit between ones that do; their rows
    do not exist, and the others are unaffected.  lse may be left out."""
    lens, chunks = [300, 50, 700, 129], [0, 50, 0, 129]
    batch, offs, q = _case(lens, chunks, 8, 2, seed=480)
    out, lse, ws = cadkv.prefill_attention(
        q.cuda(), torch.from_numpy(offs).cuda(), batch.k_pages.cuda(), batch.v_pages.cuda(),
        torch.from_numpy(batch.block_table).cuda(), torch.from_numpy(batch.context_lens).cuda(),
        want_lse=False)
    torch.cuda.synchronize()
    assert lse is None and cadkv.prefill_attention_status(ws) == 0
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(out, None, ref, ref_lse, "prefill with empty chunks, no lse")


def test_prefill_empty_job():
    batch, offs, q = _case([40, 60], [0, 0], 4, 1, seed=485)
    out, lse, ws = _run(batch, offs, q)
    assert out.shape[0] == 0 and cadkv.prefill_attention_status(ws) == 0


def test_prefill_repeat_calls_bit_identical():
    """Split items merge their pieces in piece order, whichever CTA finishes
    last: two calls give the same bits."""
    lens, chunks = [20000, 9000], [64, 300]
    batch, offs, q = _case(lens, chunks, 8, 2, seed=490)
    a_out, a_lse, _ = _run(batch, offs, q)
    b_out, b_lse, _ = _run(batch, offs, q)
    assert torch.equal(a_out, b_out) and torch.equal(a_lse, b_lse)
    ref, ref_lse = _oracle(batch, offs, q)
    assert_close(a_out, a_lse, ref, ref_lse, "prefill repeat")
