"""A KV pool that the library allocates itself (kv_pool_create with no layer
arrays), through the C ABI: the pool reports its geometry and layer pointers,
staged rows loaded into it come back bit for bit, and decode attention over
each of its layers matches the fp64 oracle."""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300.workloads import bf16_bits, scatter_block_table
from _gpu_util import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def test_library_owned_pool_load_stage_and_decode():
    lib = cadkv.library()
    layers, hkv, hq, d = 2, 2, 8, 128
    lens = np.array([37, 200, 1, 160, 0, 77], dtype=np.int32)
    batch = len(lens)
    pages = -(-lens.astype(np.int64) // 16)
    max_pages = int(pages.max())
    rng = np.random.Generator(np.random.PCG64(4242))
    table, num_pages = scatter_block_table(lens, 16, max_pages, int(pages.sum()) + 5, rng)

    handle = ctypes.c_void_p()
    assert lib.kv_pool_create(ctypes.byref(handle), layers, num_pages, 16, hkv, d, None, None) == 0
    try:
        geo = [ctypes.c_int(-1) for _ in range(5)]
        assert lib.kv_pool_geometry(handle, *[ctypes.byref(g) for g in geo]) == 0
        assert [g.value for g in geo] == [layers, num_pages, 16, hkv, d]
        k_ptr, v_ptr = ctypes.c_void_p(), ctypes.c_void_p()
        assert lib.kv_pool_layer(handle, layers, ctypes.byref(k_ptr), ctypes.byref(v_ptr)) != 0

        stream = torch.cuda.current_stream()
        s = stream.cuda_stream
        bt = torch.from_numpy(table).cuda()
        cl = torch.from_numpy(lens).cuda()
        ws = torch.empty(max(int(lib.kv_prefix_stage_workspace_size(batch)), 1),
                         dtype=torch.uint8, device="cuda")
        # packed staged rows [L][K|V][Hkv][n_b][D] per trajectory, N(0,1) values
        g = torch.Generator().manual_seed(4243)
        rows = torch.randn(int(lens.sum()) * layers * 2 * hkv * d, generator=g).to(torch.bfloat16)
        rows_gpu = rows.cuda()
        assert lib.kv_prefix_load(handle, bt.data_ptr(), max_pages, cl.data_ptr(), batch, 0, layers,
                                  rows_gpu.data_ptr(), None, ws.data_ptr(), ws.numel(), s) == 0
        back = torch.full_like(rows_gpu, float("nan"))
        assert lib.kv_prefix_stage(handle, bt.data_ptr(), max_pages, cl.data_ptr(), batch, 0, layers,
                                   back.data_ptr(), None, ws.data_ptr(), ws.numel(), s) == 0
        torch.cuda.synchronize()
        assert lib.kv_prefix_stage_status(ws.data_ptr(), s) == 0
        assert torch.equal(back.view(torch.int16), rows_gpu.view(torch.int16))

        # the oracle's pool holds the same tokens (slots past n_b stay zero there)
        kpool = np.zeros((layers, num_pages, hkv, 16, d), dtype=np.uint16)
        vpool = np.zeros_like(kpool)
        oracle.prefix_load(kpool, vpool, table, lens, 0, layers, bf16_bits(rows))
        wsd = torch.empty(int(lib.decode_attention_workspace_size(batch, hq, hkv, d, max_pages)),
                          dtype=torch.uint8, device="cuda")
        for layer in range(layers):
            assert lib.kv_pool_layer(handle, layer, ctypes.byref(k_ptr), ctypes.byref(v_ptr)) == 0
            q = torch.randn((batch, hq, d), generator=torch.Generator().manual_seed(4244 + layer))
            q = q.to(torch.bfloat16)
            qg = q.cuda()
            out = torch.empty_like(qg)
            lse = torch.empty((batch, hq), dtype=torch.float32, device="cuda")
            assert lib.decode_attention(qg.data_ptr(), k_ptr.value, v_ptr.value, bt.data_ptr(),
                                        cl.data_ptr(), out.data_ptr(), lse.data_ptr(), batch, hq,
                                        hkv, d, 16, num_pages, max_pages, wsd.data_ptr(),
                                        wsd.numel(), s) == 0
            torch.cuda.synchronize()
            assert lib.decode_attention_status(wsd.data_ptr(), s) == 0
            ref, ref_lse = oracle.decode_attention(bf16_bits(q), kpool[layer], vpool[layer], table,
                                                   lens)
            assert_close(out, lse, ref, ref_lse, f"library-owned pool, layer {layer}")
    finally:
        assert lib.kv_pool_destroy(handle) == 0
