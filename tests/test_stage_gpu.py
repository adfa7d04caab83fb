"""GPU prefix staging and loading (CUDA path through the C ABI) against the
oracle: bit-exact on every element, including NaN payloads."""
import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS
from paper_2609_36899_gb300.workloads import (STAGING, bf16_bits, fill_layer_pool,
                                              make_staging_job, scatter_block_table)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def random_bits_pool(layers, num_pages, hkv, d, seed):
    g = torch.Generator().manual_seed(seed)
    x = torch.randint(-32768, 32768, (layers, num_pages, hkv, 16, d), generator=g,
                      dtype=torch.int32).to(torch.int16)
    return x.view(torch.bfloat16)


def make_case(lens, layers, hkv, d, seed, extra=3):
    lens = np.asarray(lens, dtype=np.int32)
    pages = -(-lens.astype(np.int64) // 16)
    rng = np.random.Generator(np.random.PCG64(seed))
    max_pages = max(int(pages.max(initial=0)), 1)
    table, num_pages = scatter_block_table(lens, 16, max_pages, int(pages.sum()) + extra, rng)
    kp = random_bits_pool(layers, num_pages, hkv, d, seed)
    vp = random_bits_pool(layers, num_pages, hkv, d, seed + 1)
    return lens, table, kp, vp


def to_pool(kp, vp):
    k_layers = [kp[l].cuda().contiguous() for l in range(kp.shape[0])]
    v_layers = [vp[l].cuda().contiguous() for l in range(vp.shape[0])]
    return cadkv.KVPool(k_layers, v_layers), k_layers, v_layers


def oracle_stage(kp, vp, table, lens, lb, le, offsets=None, dst=None):
    return oracle.prefix_stage(bf16_bits(kp.reshape(-1)).reshape(kp.shape),
                               bf16_bits(vp.reshape(-1)).reshape(vp.shape),
                               table, lens, lb, le, dst_offsets=offsets, dst=dst)


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("lb,le", [(0, 3), (1, 2)])
def test_stage_bit_exact(d, lb, le):
    lens, table, kp, vp = make_case([1, 15, 16, 17, 40, 0, 333], 3, 2, d, seed=d + lb)
    pool, _, _ = to_pool(kp, vp)
    size = cadkv.staged_size(lens, lb, le, 2, d)
    dst = torch.full((size + 64,), float("nan"), dtype=torch.bfloat16, device="cuda")
    dst.view(torch.int16).fill_(0x1234)
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(),
                               torch.from_numpy(lens).cuda(), lb, le, dst)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    got = bf16_bits(dst)
    ref = oracle_stage(kp, vp, table, lens, lb, le)
    np.testing.assert_array_equal(got[:size], ref)
    assert np.all(got[size:] == 0x1234)


def test_stage_explicit_offsets_keep_gaps():
    lens, table, kp, vp = make_case([9, 33, 1], 2, 2, 128, seed=21)
    pool, _, _ = to_pool(kp, vp)
    row = 2 * 2 * 2 * 128
    sizes = [int(n) * row for n in lens]
    offs = np.array([8, 8 + sizes[0] + 16, 8 + sizes[0] + 16 + sizes[1] + 24], dtype=np.int64)
    total = int(offs[-1] + sizes[-1] + 40)
    sentinel = np.full(total, 0xABCD, dtype=np.uint16)
    dst = torch.from_numpy(sentinel.view(np.int16).copy()).view(torch.bfloat16).cuda()
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(),
                               torch.from_numpy(lens).cuda(), 0, 2, dst,
                               dst_offsets=torch.from_numpy(offs).cuda())
    assert cadkv.kv_prefix_stage_status(ws) == 0
    ref = oracle_stage(kp, vp, table, lens, 0, 2, offsets=offs, dst=sentinel.copy())
    np.testing.assert_array_equal(bf16_bits(dst), ref)


def test_stage_misaligned_offset_is_reported():
    lens, table, kp, vp = make_case([9, 3], 1, 1, 64, seed=22)
    pool, _, _ = to_pool(kp, vp)
    offs = torch.tensor([0, 9 * 2 * 64 + 3], dtype=torch.int64, device="cuda")
    dst = torch.zeros(4096, dtype=torch.bfloat16, device="cuda")
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(),
                               torch.from_numpy(lens).cuda(), 0, 1, dst, dst_offsets=offs)
    assert cadkv.kv_prefix_stage_status(ws) == STATUS["CADKV_ERR_INVALID"]


def test_stage_reports_bad_page():
    lens, table, kp, vp = make_case([20, 20], 1, 1, 64, seed=23)
    pool, _, _ = to_pool(kp, vp)
    bt = torch.from_numpy(table).cuda()
    bt[0, 1] = -7
    dst = torch.zeros(cadkv.staged_size(lens, 0, 1, 1, 64), dtype=torch.bfloat16, device="cuda")
    ws = cadkv.kv_prefix_stage(pool, bt, torch.from_numpy(lens).cuda(), 0, 1, dst)
    assert cadkv.kv_prefix_stage_status(ws) == STATUS["CADKV_ERR_OOB"]


def test_load_round_trip():
    """Stage from one pool, load into a fresh pool with another page table; the
    destination holds what the oracle's load writes, and restaging gives the
    same bytes."""
    lens, table, kp, vp = make_case([21, 64, 2, 0, 100], 2, 2, 128, seed=24)
    pool, _, _ = to_pool(kp, vp)
    lens_d = torch.from_numpy(lens).cuda()
    size = cadkv.staged_size(lens, 0, 2, 2, 128)
    staged = torch.empty(size, dtype=torch.bfloat16, device="cuda")
    cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(), lens_d, 0, 2, staged)
    rng = np.random.Generator(np.random.PCG64(25))
    pages = int((-(-lens.astype(np.int64) // 16)).sum())
    table2, n2 = scatter_block_table(lens, 16, table.shape[1], pages + 4, rng)
    k2 = torch.zeros((2, n2, 2, 16, 128), dtype=torch.bfloat16)
    v2 = torch.zeros_like(k2)
    pool2, k2_layers, v2_layers = to_pool(k2, v2)
    ws = cadkv.kv_prefix_load(pool2, torch.from_numpy(table2).cuda(), lens_d, 0, 2, staged)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    ref_k = np.zeros((2, n2, 2, 16, 128), dtype=np.uint16)
    ref_v = np.zeros_like(ref_k)
    oracle.prefix_load(ref_k, ref_v, table2, lens, 0, 2, bf16_bits(staged))
    got_k = np.stack([bf16_bits(t) for t in k2_layers])
    got_v = np.stack([bf16_bits(t) for t in v2_layers])
    np.testing.assert_array_equal(got_k, ref_k)
    np.testing.assert_array_equal(got_v, ref_v)
    again = torch.empty_like(staged)
    cadkv.kv_prefix_stage(pool2, torch.from_numpy(table2).cuda(), lens_d, 0, 2, again)
    torch.cuda.synchronize()
    assert torch.equal(again.view(torch.int16), staged.view(torch.int16))


def test_stage_to_pinned_host_bit_exact():
    """Staging straight into page-locked host memory (the copy kernel writes the
    rows over the CPU-GPU link) gives the oracle's bytes and leaves the bytes
    after the rows untouched."""
    lens, table, kp, vp = make_case([1, 15, 16, 17, 40, 0, 333, 1000], 2, 8, 128, seed=26)
    pool, _, _ = to_pool(kp, vp)
    size = cadkv.staged_size(lens, 0, 2, 8, 128)
    dst = torch.empty(size + 64, dtype=torch.bfloat16, pin_memory=True)
    dst.view(torch.int16).fill_(0x1234)
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(),
                               torch.from_numpy(lens).cuda(), 0, 2, dst)
    assert cadkv.kv_prefix_stage_status(ws) == 0  # synchronises the stream
    got = bf16_bits(dst)
    np.testing.assert_array_equal(got[:size], oracle_stage(kp, vp, table, lens, 0, 2))
    assert np.all(got[size:] == 0x1234)


def test_load_from_pinned_host_round_trip():
    """Rows kept in page-locked host memory load into a fresh pool (another page
    table) exactly as the oracle's load writes them."""
    lens, table, kp, vp = make_case([21, 64, 2, 0, 100], 2, 2, 128, seed=27)
    pool, _, _ = to_pool(kp, vp)
    lens_d = torch.from_numpy(lens).cuda()
    staged = torch.empty(cadkv.staged_size(lens, 0, 2, 2, 128), dtype=torch.bfloat16,
                         pin_memory=True)
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(table).cuda(), lens_d, 0, 2, staged)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    rng = np.random.Generator(np.random.PCG64(28))
    pages = int((-(-lens.astype(np.int64) // 16)).sum())
    table2, n2 = scatter_block_table(lens, 16, table.shape[1], pages + 4, rng)
    k2 = torch.zeros((2, n2, 2, 16, 128), dtype=torch.bfloat16)
    pool2, k2_layers, v2_layers = to_pool(k2, torch.zeros_like(k2))
    ws = cadkv.kv_prefix_load(pool2, torch.from_numpy(table2).cuda(), lens_d, 0, 2, staged)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    ref_k = np.zeros((2, n2, 2, 16, 128), dtype=np.uint16)
    ref_v = np.zeros_like(ref_k)
    oracle.prefix_load(ref_k, ref_v, table2, lens, 0, 2, bf16_bits(staged))
    np.testing.assert_array_equal(np.stack([bf16_bits(t) for t in k2_layers]), ref_k)
    np.testing.assert_array_equal(np.stack([bf16_bits(t) for t in v2_layers]), ref_v)


def test_stage_refuses_pageable_host_rows():
    """Host rows that are not page-locked are refused before anything launches,
    by the binding and by the C ABI itself."""
    import ctypes
    lens, table, kp, vp = make_case([20], 1, 1, 64, seed=29)
    pool, _, _ = to_pool(kp, vp)
    bt = torch.from_numpy(table).cuda()
    cl = torch.from_numpy(lens).cuda()
    dst = torch.zeros(cadkv.staged_size(lens, 0, 1, 1, 64) + 64, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        cadkv.kv_prefix_stage(pool, bt, cl, 0, 1, dst)
    ws = torch.empty(cadkv.kv_prefix_stage_workspace_size(1), dtype=torch.uint8, device="cuda")
    P = ctypes.c_void_p
    rc = cadkv.library().kv_prefix_stage(pool.handle, P(bt.data_ptr()), bt.shape[1],
                                         P(cl.data_ptr()), 1, 0, 1, P(dst.data_ptr()), None,
                                         P(ws.data_ptr()), ws.numel(), None)
    assert rc == STATUS["CADKV_ERR_INVALID"]
    assert torch.count_nonzero(dst.view(torch.int16)) == 0


def test_full_size_staging_sampled():
    """All 64 trajectories of the staging workload (lengths 8K..64K tokens,
    8 KV heads, D = 128) for two layers; every staged row of four sampled
    trajectories is compared bit for bit with the oracle's gather."""
    job = make_staging_job(STAGING)
    layers = 2
    k_layers = [torch.empty((job.num_pages, 8, 16, 128), dtype=torch.bfloat16, device="cuda")
                for _ in range(layers)]
    v_layers = [torch.empty_like(k_layers[0]) for _ in range(layers)]
    for l in range(layers):
        fill_layer_pool(k_layers[l], v_layers[l], STAGING.seed, l)
    pool = cadkv.KVPool(k_layers, v_layers)
    lens = job.context_lens
    size = cadkv.staged_size(lens, 0, layers, 8, 128)
    dst = torch.empty(size, dtype=torch.bfloat16, device="cuda")
    ws = cadkv.kv_prefix_stage(pool, torch.from_numpy(job.block_table).cuda(),
                               torch.from_numpy(lens).cuda(), 0, layers, dst)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    row = layers * 2 * 8 * 128
    starts = np.concatenate([[0], np.cumsum(lens.astype(np.int64) * row)])
    for b in (0, int(np.argmax(lens)), int(np.argmin(lens)), 37):
        p = -(-int(lens[b]) // 16)
        phys = torch.from_numpy(job.block_table[b, :p].astype(np.int64)).cuda()
        kp = torch.stack([k_layers[l].index_select(0, phys) for l in range(layers)]).cpu()
        vp = torch.stack([v_layers[l].index_select(0, phys) for l in range(layers)]).cpu()
        ref = oracle_stage(kp, vp, np.arange(p, dtype=np.int32)[None], lens[b:b + 1], 0, layers)
        got = bf16_bits(dst[int(starts[b]):int(starts[b + 1])])
        np.testing.assert_array_equal(got, ref)
    del dst, k_layers, v_layers, pool
    torch.cuda.empty_cache()
