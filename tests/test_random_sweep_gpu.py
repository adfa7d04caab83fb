"""Seeded random sweep over the configuration space of every kernel, each case
compared element by element with the fp64 oracle (bit-exact for the pool and
the staged rows).

The fixed-shape tests pin chosen corners; this sweep draws shapes nobody chose:
head_dim 64 or 128, 1-8 KV heads, GQA groups 1-8, batches of 1-400, lengths
drawn from uniform (with zeros), lognormal, "one long trajectory among short
ones" and all-equal distributions, tables wider than needed, forced or automatic
slicing, K scaled by 0.5-2.  Each case's draw depends only on its index, so a
failure names a reproducible case.  Sizes are bounded so that the oracle of one
case finishes in about a second.

Attention outputs are held to 1e-2, raised per element to the bound of the
kernels' own rounding where that is larger (rows over a handful of keys with
large values; see assert_close_bounded); the LSE to 1e-3 relative.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300.workloads import bf16_bits, scatter_block_table
from _gpu_util import abs_bits, assert_close_bounded, gpu_decode, make_batch

pytestmark = pytest.mark.gpu

DECODE_CASES = 64
APPEND_CASES = 16
PREFILL_CASES = 32
STAGE_CASES = 32


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def _lengths(rng, batch, kind, cap):
    if kind == 0:      # uniform, zeros included
        lens = rng.integers(0, cap + 1, batch)
    elif kind == 1:    # lognormal, heavy-tailed
        lens = np.clip(np.round(cap / 8 * np.exp(rng.normal(0.0, 1.2, batch))), 1, cap)
    elif kind == 2:    # one long trajectory among short ones
        lens = rng.integers(1, 64, batch)
        lens[rng.integers(0, batch)] = rng.integers(cap // 2, cap + 1)
    else:              # all equal
        lens = np.full(batch, rng.integers(1, cap + 1))
    return lens.astype(np.int64)


def _bounded(lens, budget):
    """Scale lengths down so that their sum stays within `budget`."""
    total = int(lens.sum())
    if total > budget:
        lens = np.floor(lens * (budget / total)).astype(np.int64)
    return lens.astype(np.int32)


def _decode_shape(rng):
    d = int(rng.choice([64, 128]))
    hkv = int(rng.choice([1, 2, 4, 8]))
    g = int(rng.integers(1, 9))
    batch = max(1, int(np.exp(rng.uniform(0.0, np.log(400.0)))))
    return d, hkv, g, batch


@pytest.mark.parametrize("case", range(DECODE_CASES))
def test_decode_random_case(case):
    rng = np.random.Generator(np.random.PCG64(7000 + case))
    d, hkv, g, batch = _decode_shape(rng)
    lens = _lengths(rng, batch, int(rng.integers(0, 4)), int(rng.choice([300, 3000, 30000])))
    lens = _bounded(lens, 3_000_000 // (g * hkv))
    need = int((-(-lens.astype(np.int64) // 16)).max(initial=0))
    max_pages = max(need, 1) + int(rng.integers(0, 3))
    slice_pages = 0 if rng.random() < 0.5 else int(rng.integers(1, 65))
    k_scale = float(rng.choice([0.5, 1.0, 2.0]))
    b = make_batch(lens, g * hkv, hkv, d, seed=7100 + case,
                   extra_pages=int(rng.integers(0, 9)), max_pages=max_pages, k_scale=k_scale)
    out, lse = gpu_decode(b, slice_pages=slice_pages)
    qb, kb, vb = bf16_bits(b.q), bf16_bits(b.k_pages), bf16_bits(b.v_pages)
    ref, ref_lse = oracle.decode_attention(qb, kb, vb, b.block_table, b.context_lens)
    absv, _ = oracle.decode_attention(qb, kb, abs_bits(vb), b.block_table, b.context_lens)
    assert_close_bounded(out, lse, ref, ref_lse, absv,
                         f"decode case {case}: B={batch} G={g} Hkv={hkv} D={d} "
                         f"slice_pages={slice_pages} sum_n={int(lens.sum())}")


@pytest.mark.parametrize("case", range(APPEND_CASES))
def test_append_random_case(case):
    rng = np.random.Generator(np.random.PCG64(7200 + case))
    d, hkv, g, batch = _decode_shape(rng)
    lens = _lengths(rng, batch, int(rng.integers(0, 4)), int(rng.choice([300, 3000])))
    lens = _bounded(lens, 1_000_000 // (g * hkv))
    b = make_batch(lens, g * hkv, hkv, d, seed=7300 + case)   # NaN in the new slots
    gen = torch.Generator().manual_seed(7400 + case)
    k_new = torch.randn((batch, hkv, d), generator=gen).to(torch.bfloat16)
    v_new = torch.randn((batch, hkv, d), generator=gen).to(torch.bfloat16)
    kp = bf16_bits(b.k_pages).copy()
    vp = bf16_bits(b.v_pages).copy()
    oracle.kv_append(kp, vp, bf16_bits(k_new), bf16_bits(v_new), b.block_table, b.context_lens)
    k_dev, v_dev = b.k_pages.cuda(), b.v_pages.cuda()
    out, lse = cadkv.decode_attention_append(
        b.q.cuda(), k_new.cuda(), v_new.cuda(), k_dev, v_dev,
        torch.from_numpy(b.block_table).cuda(), torch.from_numpy(b.context_lens).cuda())
    torch.cuda.synchronize()
    np.testing.assert_array_equal(bf16_bits(k_dev), kp)
    np.testing.assert_array_equal(bf16_bits(v_dev), vp)
    ref, ref_lse = oracle.decode_attention(bf16_bits(b.q), kp, vp, b.block_table,
                                           b.context_lens)
    absv, _ = oracle.decode_attention(bf16_bits(b.q), kp, abs_bits(vp), b.block_table,
                                      b.context_lens)
    assert_close_bounded(out, lse, ref, ref_lse, absv,
                         f"append case {case}: B={batch} G={g} Hkv={hkv} D={d}")


@pytest.mark.parametrize("case", range(PREFILL_CASES))
def test_prefill_random_case(case):
    rng = np.random.Generator(np.random.PCG64(7500 + case))
    hkv = int(rng.choice([1, 2, 4, 8]))
    g = int(rng.integers(1, 9))
    hq = g * hkv
    batch = int(rng.integers(1, 41))
    lens = np.maximum(_lengths(rng, batch, int(rng.integers(0, 4)), 3000), 1)
    chunks = np.minimum(lens, rng.integers(0, 600, batch))
    # bound the oracle's work: sum of chunk x context x query heads
    work = int((chunks * lens).sum()) * hq
    if work > 20_000_000:
        f = np.sqrt(20_000_000 / work)
        lens = np.maximum(np.floor(lens * f), 1).astype(np.int64)
        chunks = np.minimum(lens, np.floor(chunks * f).astype(np.int64))
    lens = lens.astype(np.int32)
    b = make_batch(lens, hq, hkv, 128, seed=7600 + case)
    offs = np.concatenate([[0], np.cumsum(chunks)]).astype(np.int64)
    gen = torch.Generator().manual_seed(7700 + case)
    q = torch.randn((int(offs[-1]), hq, 128), generator=gen).to(torch.bfloat16)
    out, lse, ws = cadkv.prefill_attention(
        q.cuda(), torch.from_numpy(offs).cuda(), b.k_pages.cuda(), b.v_pages.cuda(),
        torch.from_numpy(b.block_table).cuda(), torch.from_numpy(b.context_lens).cuda())
    torch.cuda.synchronize()
    assert cadkv.prefill_attention_status(ws) == 0
    qb, kb, vb = bf16_bits(q), bf16_bits(b.k_pages), bf16_bits(b.v_pages)
    ref, ref_lse = oracle.prefill_attention(qb, offs, kb, vb, b.block_table, b.context_lens)
    absv, _ = oracle.prefill_attention(qb, offs, kb, abs_bits(vb), b.block_table,
                                       b.context_lens)
    assert_close_bounded(out, lse, ref, ref_lse, absv,
                         f"prefill case {case}: B={batch} G={g} Hkv={hkv} rows={int(offs[-1])}")


def _pool_bits(layers, num_pages, hkv, d, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randint(-32768, 32768, (layers, num_pages, hkv, 16, d), generator=g,
                      dtype=torch.int32).to(torch.int16)
    return x.view(torch.bfloat16)


@pytest.mark.parametrize("case", range(STAGE_CASES))
def test_stage_and_load_random_case(case):
    rng = np.random.Generator(np.random.PCG64(7800 + case))
    d = int(rng.choice([64, 128]))
    hkv = int(rng.choice([1, 2, 4, 8]))
    layers = int(rng.integers(1, 5))
    lb = int(rng.integers(0, layers))
    le = int(rng.integers(lb + 1, layers + 1))
    batch = max(1, int(np.exp(rng.uniform(0.0, np.log(300.0)))))
    lens = _lengths(rng, batch, int(rng.integers(0, 4)), 2000)
    row_bytes = (le - lb) * 2 * hkv * d * 2
    lens = _bounded(lens, 200_000_000 // row_bytes)
    pages = -(-lens.astype(np.int64) // 16)
    max_pages = max(int(pages.max(initial=0)), 1) + int(rng.integers(0, 3))
    table, num_pages = scatter_block_table(lens, 16, max_pages,
                                           int(pages.sum()) + int(rng.integers(1, 6)), rng)
    kp = _pool_bits(layers, num_pages, hkv, d, 7900 + case)
    vp = _pool_bits(layers, num_pages, hkv, d, 8000 + case)
    k_layers = [kp[l].cuda().contiguous() for l in range(layers)]
    v_layers = [vp[l].cuda().contiguous() for l in range(layers)]
    pool = cadkv.KVPool(k_layers, v_layers)
    bt, cl = torch.from_numpy(table).cuda(), torch.from_numpy(lens).cuda()
    kbits = bf16_bits(kp.reshape(-1)).reshape(kp.shape)
    vbits = bf16_bits(vp.reshape(-1)).reshape(vp.shape)

    # explicit offsets with 16-byte-aligned gaps in half of the cases
    rows = lens.astype(np.int64) * (le - lb) * 2 * hkv * d
    offsets = None
    total = int(rows.sum())
    if rng.random() < 0.5:
        gaps = 8 * rng.integers(0, 5, batch)
        offsets = np.concatenate([[0], np.cumsum(rows + gaps)[:-1]]).astype(np.int64) + gaps[0]
        total = int(offsets[-1] + rows[-1]) + 8
    sentinel = np.full(total + 16, 0x5A5A, dtype=np.uint16)
    dst = torch.from_numpy(sentinel.view(np.int16).copy()).view(torch.bfloat16).cuda()
    ws = cadkv.kv_prefix_stage(pool, bt, cl, lb, le, dst,
                               dst_offsets=None if offsets is None
                               else torch.from_numpy(offsets).cuda())
    assert cadkv.kv_prefix_stage_status(ws) == 0
    ref = oracle.prefix_stage(kbits, vbits, table, lens, lb, le, dst_offsets=offsets,
                              dst=sentinel.copy())
    got = bf16_bits(dst)
    np.testing.assert_array_equal(got[:len(ref)], ref,
                                  err_msg=f"stage case {case}: B={batch} Hkv={hkv} D={d} "
                                          f"layers [{lb}, {le})")

    # load the rows into another pool under another page table
    table2, n2 = scatter_block_table(lens, 16, max_pages, int(pages.sum()) + 2, rng)
    k2 = [torch.zeros((n2, hkv, 16, d), dtype=torch.bfloat16, device="cuda")
          for _ in range(layers)]
    v2 = [torch.zeros_like(t) for t in k2]
    pool2 = cadkv.KVPool(k2, v2)
    ws = cadkv.kv_prefix_load(pool2, torch.from_numpy(table2).cuda(), cl, lb, le, dst,
                              src_offsets=None if offsets is None
                              else torch.from_numpy(offsets).cuda())
    assert cadkv.kv_prefix_stage_status(ws) == 0
    ref_k = np.zeros((layers, n2, hkv, 16, d), dtype=np.uint16)
    ref_v = np.zeros_like(ref_k)
    oracle.prefix_load(ref_k, ref_v, table2, lens, lb, le, got, src_offsets=offsets)
    np.testing.assert_array_equal(np.stack([bf16_bits(t) for t in k2]), ref_k)
    np.testing.assert_array_equal(np.stack([bf16_bits(t) for t in v2]), ref_v)
