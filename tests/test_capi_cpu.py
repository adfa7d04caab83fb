"""The C-ABI library loads and exports every symbol include/cadkv.h declares,
and host-side argument validation answers with the documented status codes.
None of these calls reaches the GPU."""
import ctypes

import pytest

import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS

NULL = None


@pytest.fixture(scope="module")
def lib():
    from paper_2609_36899_gb300 import build
    build.build()
    return cadkv.library()


def test_every_declared_function_is_exported(lib):
    names = cadkv.header_functions()
    assert "decode_attention" in names and "kv_prefix_stage" in names
    assert "kv_pool_create" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings(lib):
    for name, code in STATUS.items():
        text = cadkv.kv_status_string(code)
        assert text and text != "unknown status", name
    assert cadkv.kv_status_string(12345) == "unknown status"
    assert lib.cadkv_abi_version() >> 16 == 1


def _decode(lib, **over):
    args = dict(q=1 << 12, k=1 << 12, v=1 << 12, bt=1 << 12, cl=1 << 12, out=1 << 12,
                lse=None, batch=4, hq=8, hkv=2, d=64, page=16, num_pages=128, max_pages=64,
                ws=1 << 12, ws_bytes=1 << 30)
    args.update(over)
    P = ctypes.c_void_p
    return lib.decode_attention(P(args["q"]), P(args["k"]), P(args["v"]), P(args["bt"]),
                                P(args["cl"]), P(args["out"]), P(args["lse"]), args["batch"],
                                args["hq"], args["hkv"], args["d"], args["page"],
                                args["num_pages"], args["max_pages"], P(args["ws"]),
                                args["ws_bytes"], None)


@pytest.mark.parametrize("over,code", [
    (dict(q=None), "CADKV_ERR_INVALID"),
    (dict(out=None), "CADKV_ERR_INVALID"),
    (dict(cl=None), "CADKV_ERR_INVALID"),
    (dict(q=(1 << 12) + 2), "CADKV_ERR_INVALID"),           # misaligned
    (dict(hq=6, hkv=4), "CADKV_ERR_SHAPE"),                 # Hq % Hkv != 0
    (dict(hq=32, hkv=2), "CADKV_ERR_UNSUPPORTED"),          # G = 16
    (dict(d=96), "CADKV_ERR_UNSUPPORTED"),
    (dict(page=32), "CADKV_ERR_UNSUPPORTED"),
    (dict(batch=-1), "CADKV_ERR_SHAPE"),
    (dict(num_pages=0), "CADKV_ERR_SHAPE"),
    (dict(max_pages=-3), "CADKV_ERR_SHAPE"),
    (dict(max_pages=1 << 27), "CADKV_ERR_SHAPE"),            # 16 * max_pages tokens overflow int32
    (dict(num_pages=1 << 30), "CADKV_ERR_UNSUPPORTED"),      # page-head rows overflow int32
])
def test_decode_attention_rejects_on_host(lib, over, code):
    assert _decode(lib, **over) == STATUS[code]


def test_empty_batch_is_a_no_op(lib):
    assert _decode(lib, batch=0, q=None, out=None) == 0


def test_workspace_size_rejects_bad_shapes(lib):
    assert lib.decode_attention_workspace_size(4, 6, 4, 64, 10) == 0
    assert lib.decode_attention_workspace_size(4, 8, 2, 96, 10) == 0
    assert lib.kv_prefix_stage_workspace_size(-1) == 0
    assert lib.kv_prefix_stage_workspace_size(64) > 64 * 3 * 8


def test_pool_create_rejects_on_host(lib):
    h = ctypes.c_void_p()
    P = ctypes.c_void_p
    assert lib.kv_pool_create(None, 1, 8, 16, 2, 64, None, None) == STATUS["CADKV_ERR_INVALID"]
    assert lib.kv_pool_create(ctypes.byref(h), 0, 8, 16, 2, 64, None, None) == STATUS["CADKV_ERR_SHAPE"]
    assert lib.kv_pool_create(ctypes.byref(h), 1, 8, 8, 2, 64, None, None) == STATUS["CADKV_ERR_UNSUPPORTED"]
    assert lib.kv_pool_create(ctypes.byref(h), 1, 8, 16, 2, 80, None, None) == STATUS["CADKV_ERR_UNSUPPORTED"]
    arr = (ctypes.c_void_p * 1)(1 << 12)
    assert lib.kv_pool_create(ctypes.byref(h), 1, 8, 16, 2, 64, ctypes.cast(arr, P), None) == \
        STATUS["CADKV_ERR_INVALID"]
    bad = (ctypes.c_void_p * 1)((1 << 12) + 8)
    assert lib.kv_pool_create(ctypes.byref(h), 1, 8, 16, 2, 64, ctypes.cast(bad, P),
                              ctypes.cast(bad, P)) == STATUS["CADKV_ERR_INVALID"]
    assert lib.kv_pool_destroy(None) == 0


def test_stage_rejects_null_pool(lib):
    P = ctypes.c_void_p
    assert lib.kv_prefix_stage(None, P(1 << 12), 4, P(1 << 12), 2, 0, 1, P(1 << 12), None,
                               P(1 << 12), 1 << 20, None) == STATUS["CADKV_ERR_INVALID"]


def test_read_probe_rejects_on_host(lib):
    P = ctypes.c_void_p
    assert lib.cadkv_hbm_read_probe(None, 16, P(1 << 12), None) == STATUS["CADKV_ERR_INVALID"]
    assert lib.cadkv_hbm_read_probe(P(1 << 12), 15, P(1 << 12), None) == STATUS["CADKV_ERR_INVALID"]
    assert lib.cadkv_hbm_read_probe(P((1 << 12) + 4), 16, P(1 << 12), None) == \
        STATUS["CADKV_ERR_INVALID"]
    assert lib.cadkv_hbm_read_probe(P(1 << 12), 0, P(1 << 12), None) == 0


def test_prefill_rejects_on_host(lib):
    P = ctypes.c_void_p
    a = P(1 << 12)

    def call(**over):
        args = dict(q=a, offs=a, k=a, v=a, bt=a, cl=a, out=a, batch=2, total=8, hq=8, hkv=2,
                    d=128, page=16, num_pages=4, max_pages=4)
        args.update(over)
        return lib.prefill_attention(args["q"], args["offs"], args["k"], args["v"], args["bt"],
                                     args["cl"], args["out"], None, args["batch"], args["total"],
                                     args["hq"], args["hkv"], args["d"], args["page"],
                                     args["num_pages"], args["max_pages"], a, 1 << 20, None)
    assert call(d=64) == STATUS["CADKV_ERR_UNSUPPORTED"]
    assert call(hq=18, hkv=2) == STATUS["CADKV_ERR_UNSUPPORTED"]     # G = 9 > 8
    assert call(hq=6, hkv=4) == STATUS["CADKV_ERR_SHAPE"]
    assert call(q=None) == STATUS["CADKV_ERR_INVALID"]
    assert call(offs=P((1 << 12) + 4)) == STATUS["CADKV_ERR_INVALID"]
    assert call(total=0) == 0
    assert call(num_pages=1 << 30) == STATUS["CADKV_ERR_UNSUPPORTED"]
    assert call(max_pages=1 << 27) == STATUS["CADKV_ERR_UNSUPPORTED"]
