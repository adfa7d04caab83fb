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


def test_stage_and_load_many_trajectories():
    """1,500 trajectories (the planner's prefix sums run over several 1,024-wide
    rounds), lengths 0..200, 2 layers: staging bit-exact against the oracle, and
    loading the rows back into a cleared pool restores every used slot."""
    rng = np.random.Generator(np.random.PCG64(31))
    lens = rng.integers(0, 201, 1500)
    lens, table, kp, vp = make_case(lens.tolist(), 2, 2, 64, seed=32)
    pool, k_layers, v_layers = to_pool(kp, vp)
    bt, cl = torch.from_numpy(table).cuda(), torch.from_numpy(lens).cuda()
    size = cadkv.staged_size(lens, 0, 2, 2, 64)
    dst = torch.empty(size, dtype=torch.bfloat16, device="cuda")
    ws = cadkv.kv_prefix_stage(pool, bt, cl, 0, 2, dst)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    np.testing.assert_array_equal(bf16_bits(dst), oracle_stage(kp, vp, table, lens, 0, 2))
    for t in k_layers + v_layers:
        t.view(torch.int16).fill_(0)
    cadkv.kv_prefix_load(pool, bt, cl, 0, 2, dst, workspace=ws)
    assert cadkv.kv_prefix_stage_status(ws) == 0
    kz = torch.zeros_like(kp)
    vz = torch.zeros_like(vp)
    kl, vl = oracle.prefix_load(bf16_bits(kz.reshape(-1)).reshape(kz.shape).copy(),
                                bf16_bits(vz.reshape(-1)).reshape(vz.shape).copy(),
                                table, lens, 0, 2, bf16_bits(dst))
    for l in range(2):
        np.testing.assert_array_equal(bf16_bits(k_layers[l]), kl[l])
        np.testing.assert_array_equal(bf16_bits(v_layers[l]), vl[l])


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


def test_staging_whole_job_every_chunk_bit_exact():
    """The whole staging job: all 64 trajectories (8K..64K tokens) x 48 layers,
    8 KV heads, D = 128 -- ~464 GB per copy, more than HBM -- staged in chunks of
    layers as the bench runs it (each chunk's pool refilled from the per-layer
    seeds).  Every staged row of every layer of every trajectory is compared bit
    for bit with the oracle's gather of the same layer."""
    job = make_staging_job(STAGING)
    hkv, d, total = STAGING.num_kv_heads, STAGING.head_dim, STAGING.num_layers
    lens = job.context_lens
    rows_layer = cadkv.staged_size(lens, 0, 1, hkv, d)           # elements per layer
    pool_layer_bytes = 2 * job.num_pages * hkv * 16 * d * 2
    torch.cuda.empty_cache()
    free, _ = torch.cuda.mem_get_info()
    lc = next(c for c in (6, 4, 3, 2, 1)
              if c * (pool_layer_bytes + 2 * rows_layer) + 2 * rows_layer <= 0.8 * free)
    k_layers = [torch.empty((job.num_pages, hkv, 16, d), dtype=torch.bfloat16, device="cuda")
                for _ in range(lc)]
    v_layers = [torch.empty_like(k_layers[0]) for _ in range(lc)]
    pool = cadkv.KVPool(k_layers, v_layers)
    bt = torch.from_numpy(job.block_table).cuda()
    cl = torch.from_numpy(lens).cuda()
    dst = torch.empty(rows_layer * lc, dtype=torch.bfloat16, device="cuda")
    # host buffers (page-locked, reused for every layer) and the oracle's rows on the device
    k_host = torch.empty(k_layers[0].shape, dtype=torch.bfloat16, pin_memory=True)
    v_host = torch.empty(k_layers[0].shape, dtype=torch.bfloat16, pin_memory=True)
    ref_host = torch.empty(rows_layer, dtype=torch.bfloat16, pin_memory=True)
    ref_dev = torch.empty(rows_layer, dtype=torch.bfloat16, device="cuda")
    as_u16 = lambda t: t.view(torch.int16).numpy().view(np.uint16)   # noqa: E731
    per_b = lens.astype(np.int64) * 2 * hkv * d                 # elements of one layer
    ref_starts = np.concatenate([[0], np.cumsum(per_b)])
    ws = None
    checked = 0
    for c in range(total // lc):
        for i in range(lc):
            fill_layer_pool(k_layers[i], v_layers[i], STAGING.seed, c * lc + i)
        ws = cadkv.kv_prefix_stage(pool, bt, cl, 0, lc, dst, workspace=ws)
        assert cadkv.kv_prefix_stage_status(ws) == 0
        got = dst.view(torch.int16)
        for i in range(lc):
            k_host.copy_(k_layers[i])
            v_host.copy_(v_layers[i])
            oracle.prefix_stage(as_u16(k_host)[None], as_u16(v_host)[None], job.block_table,
                                lens, 0, 1, dst=as_u16(ref_host))
            ref_dev.copy_(ref_host)
            ref = ref_dev.view(torch.int16)
            for b in range(len(lens)):
                g0 = lc * int(ref_starts[b]) + i * int(per_b[b])
                if not torch.equal(got[g0:g0 + int(per_b[b])],
                                   ref[int(ref_starts[b]):int(ref_starts[b + 1])]):
                    raise AssertionError(f"layer {c * lc + i}, trajectory {b}: not bit-exact")
            checked += 1
    assert checked == total
    del dst, k_layers, v_layers, pool, ref_dev
    torch.cuda.empty_cache()
