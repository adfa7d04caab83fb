"""decode_attention_noalloc: decode attention for callers that cannot allocate
device memory when they call it (for example a serving engine that reserved
nearly all HBM for its KV cache up front, or a plugin with no access to its
host framework's allocator).  It uses the library's built-in scratch array
instead of a caller workspace.

Called here through the C ABI (ctypes, no binding wrapper) and compared,
within the tolerances of the other parity tests, with the fp64 oracle and with
decode_attention (caller workspace) on the same inputs, on two calls in a row,
and after other problems that left their contents in the shared scratch.  This
file is collected last so that a failure here never hides another test's
result.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS
from paper_2609_36899_gb300.workloads import bf16_bits

pytestmark = pytest.mark.gpu

OUT_ATOL = 1e-2
LSE_RTOL = 1e-3   # relative to max(|lse|, 1), as in the other parity tests


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _call_noalloc(q, k, v, bt, cl, out, lse):
    lib = cadkv.library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return lib.decode_attention_noalloc(
        _ptr(q), _ptr(k), _ptr(v), _ptr(bt), _ptr(cl), _ptr(out), _ptr(lse),
        q.shape[0], q.shape[1], k.shape[1], q.shape[2], k.shape[2], k.shape[0], bt.shape[1],
        stream)


def _inputs(lens, hq, hkv, d, seed):
    g = torch.Generator().manual_seed(seed)
    lens = np.asarray(lens, dtype=np.int32)
    pages = -(-lens.astype(np.int64) // 16)
    num_pages = int(pages.sum()) + 3
    perm = torch.randperm(num_pages, generator=g).numpy()
    max_pages = max(int(pages.max()), 1)
    table = np.full((len(lens), max_pages), -1, dtype=np.int32)
    pos = 0
    for b, p in enumerate(pages):
        table[b, :p] = perm[pos:pos + p]
        pos += p
    q = torch.randn((len(lens), hq, d), generator=g).to(torch.bfloat16).cuda()
    k = torch.randn((num_pages, hkv, 16, d), generator=g).to(torch.bfloat16).cuda()
    v = torch.randn((num_pages, hkv, 16, d), generator=g).to(torch.bfloat16).cuda()
    return q, k, v, torch.from_numpy(table).cuda(), torch.from_numpy(lens).cuda()


def _compare(out, lse, ref_out, ref_lse):
    err = (out.float() - ref_out.float()).abs().max().item()
    assert err <= OUT_ATOL, err
    fin = torch.isfinite(ref_lse)
    assert torch.equal(torch.isneginf(lse), torch.isneginf(ref_lse))
    rel = ((lse[fin] - ref_lse[fin]).abs() / ref_lse[fin].abs().clamp(min=1.0)).max().item()
    assert rel <= LSE_RTOL, rel


def _compare_oracle(out, lse, q, k, v, bt, cl):
    """Against the fp64 oracle on the same bf16 bits."""
    ref, ref_lse = oracle.decode_attention(bf16_bits(q), bf16_bits(k), bf16_bits(v),
                                           bt.cpu().numpy(), cl.cpu().numpy())
    o = out.float().cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(o))
    err = np.abs(o - ref).max(initial=0.0)
    assert err <= OUT_ATOL, err
    l = lse.cpu().numpy().astype(np.float64)
    inf_ref = np.isneginf(ref_lse)
    assert np.array_equal(np.isneginf(l), inf_ref)
    fin = ~inf_ref
    if fin.any():
        rel = (np.abs(l[fin] - ref_lse[fin]) / np.maximum(np.abs(ref_lse[fin]), 1.0)).max()
        assert rel <= LSE_RTOL, rel


@pytest.mark.parametrize("lens,hq,hkv,d", [
    ([17, 64, 250, 1000], 8, 2, 64),
    ([0, 1, 300, 4100, 12000, 33], 64, 8, 128),
])
def test_noalloc_matches_workspace_entry_point_twice(lens, hq, hkv, d):
    q, k, v, bt, cl = _inputs(lens, hq, hkv, d, seed=len(lens) * 7 + d)
    ref_out, ref_lse = cadkv.decode_attention(q, k, v, bt, cl)
    for _ in range(2):   # the scratch keeps the previous call's contents
        out = torch.full_like(q, float("nan"))
        lse = torch.full((q.shape[0], hq), float("nan"), dtype=torch.float32, device="cuda")
        assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
        torch.cuda.synchronize()
        _compare(out, lse, ref_out, ref_lse)
        _compare_oracle(out, lse, q, k, v, bt, cl)


def test_noalloc_after_a_different_problem():
    """A second, different problem on the shared scratch still matches."""
    a = _inputs([5000, 40], 32, 8, 128, seed=3)
    b = _inputs([70, 900, 2, 16], 8, 1, 64, seed=4)
    for q, k, v, bt, cl in (a, b, a):
        ref_out, ref_lse = cadkv.decode_attention(q, k, v, bt, cl)
        out = torch.empty_like(q)
        lse = torch.empty((q.shape[0], q.shape[1]), dtype=torch.float32, device="cuda")
        assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
        torch.cuda.synchronize()
        _compare(out, lse, ref_out, ref_lse)
        _compare_oracle(out, lse, q, k, v, bt, cl)


def test_noalloc_many_partials_after_a_bigger_problem():
    """A long trajectory next to short ones is cut into many slices, so its
    (trajectory, KV head) units go through several partial slots and arrival
    counters of the shared scratch; it runs right after a bigger problem left
    its own partials and counters there, and twice in a row, each time against
    the oracle."""
    big = _inputs([40000, 9000, 300, 77, 20000, 5, 60000, 1200], 64, 8, 128, seed=11)
    small = _inputs([60000, 20, 33, 100, 1], 32, 8, 128, seed=12)
    for q, k, v, bt, cl in (big, small, small):
        out = torch.full_like(q, float("nan"))
        lse = torch.full((q.shape[0], q.shape[1]), float("nan"), dtype=torch.float32,
                         device="cuda")
        assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
        torch.cuda.synchronize()
        _compare_oracle(out, lse, q, k, v, bt, cl)


def test_noalloc_rejects_problems_beyond_the_scratch():
    """20,000 trajectories x 8 KV heads need far more than 32 MiB of scratch:
    rejected on the host, nothing launched."""
    batch, hq, hkv, d = 20000, 64, 8, 128
    need = cadkv.decode_attention_workspace_size(batch, hq, hkv, d, 1)
    assert need > (32 << 20)
    q = torch.zeros((batch, hq, d), dtype=torch.bfloat16, device="cuda")
    k = torch.zeros((4, hkv, 16, d), dtype=torch.bfloat16, device="cuda")
    bt = torch.zeros((batch, 1), dtype=torch.int32, device="cuda")
    cl = torch.zeros((batch,), dtype=torch.int32, device="cuda")
    out = torch.full_like(q, 7.0)
    lse = torch.empty((batch, hq), dtype=torch.float32, device="cuda")
    assert _call_noalloc(q, k, k, bt, cl, out, lse) == STATUS["CADKV_ERR_WORKSPACE"]
    torch.cuda.synchronize()
    assert torch.all(out == 7.0)   # nothing ran


def test_noalloc_status_reports_bad_input_without_faulting():
    """The status word of the last call, read through the C ABI: a block-table
    entry outside the pool is read as page 0 and flagged CADKV_ERR_OOB, a length
    beyond the table is treated as empty and flagged CADKV_ERR_SHAPE, and the
    next good call clears the word.  The untouched trajectories still match the
    oracle."""
    lib = cadkv.library()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    q, k, v, bt, cl = _inputs([40, 20, 300], 8, 2, 64, seed=21)
    out = torch.empty_like(q)
    lse = torch.empty((3, 8), dtype=torch.float32, device="cuda")
    assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
    assert lib.decode_attention_noalloc_status(stream) == 0

    good = int(bt[1, 0])
    bt[1, 0] = k.shape[0] + 5                       # outside the pool
    assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
    assert lib.decode_attention_noalloc_status(stream) == STATUS["CADKV_ERR_OOB"]
    keep = torch.tensor([0, 2], device="cuda")
    _compare_oracle(out[keep], lse[keep], q[keep], k, v, bt[keep], cl[keep])
    bt[1, 0] = good

    cl[1] = bt.shape[1] * 16 + 1                    # longer than its table row
    assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
    assert lib.decode_attention_noalloc_status(stream) == STATUS["CADKV_ERR_SHAPE"]
    assert torch.all(out[1] == 0) and torch.all(torch.isneginf(lse[1]))
    cl[1] = 20

    assert _call_noalloc(q, k, v, bt, cl, out, lse) == 0
    assert lib.decode_attention_noalloc_status(stream) == 0
    _compare_oracle(out, lse, q, k, v, bt, cl)
    # the binding's accessor reads the same word
    assert cadkv.decode_attention_noalloc_status() == 0
