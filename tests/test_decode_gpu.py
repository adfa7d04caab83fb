"""GPU parity of decode attention (CUDA path through the C ABI) against the
fp64 oracle, on the same bf16 inputs.

Sizes: the tiny workload in full; the paced / long-tail / mixed workloads at
reduced batch sizes with their length distributions, and at their full sizes
in the bench's launch configuration, every output row against the oracle;
plus ragged, empty, maximal and degenerate cases and the method's invariances.
"""
import numpy as np
import pytest
import torch

import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300 import STATUS
from paper_2609_36899_gb300.workloads import (LONG_TAIL, MIXED, PACED, TINY, DecodeBatch,
                                              bf16_bits, make_decode_batch)
from _gpu_util import (assert_close, device_tensors, full_oracle, gpu_decode, make_batch,
                       oracle_decode)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_2609_36899_gb300 import build
    build.build()


def test_tiny_workload_full():
    batch = make_decode_batch(TINY, device="cpu")
    out, lse = gpu_decode(batch)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, "tiny")


@pytest.mark.parametrize("w,bsz", [(PACED, 24), (LONG_TAIL, 2), (MIXED, 40)],
                         ids=["paced", "long_tail", "mixed"])
def test_reduced_workloads_full_oracle(w, bsz):
    batch = make_decode_batch(w, device="cpu", batch=bsz)
    out, lse = gpu_decode(batch)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, w.name)


@pytest.mark.parametrize("w", [PACED, LONG_TAIL, MIXED], ids=["paced", "long_tail", "mixed"])
def test_full_size_every_row(w):
    """Full-size batch generated on the GPU, run in the bench's launch
    configuration (automatic slicing: the mixed batch takes the dynamic-slice
    path with multi-CTA merges of its long tails), and EVERY (trajectory,
    query head) row of out and lse compared with the fp64 oracle."""
    batch = make_decode_batch(w, device="cuda")
    tensors = (batch.q, batch.k_pages, batch.v_pages,
               torch.from_numpy(batch.block_table).cuda(),
               torch.from_numpy(batch.context_lens).cuda())
    out, lse = gpu_decode(batch, tensors=tensors)
    ref, ref_lse = full_oracle(batch)
    assert ref.shape == tuple(out.shape)
    assert_close(out, lse, ref, ref_lse, f"{w.name}, all {len(batch.context_lens)} trajectories")
    del batch, tensors
    torch.cuda.empty_cache()


def test_mixed_full_size_plan_then_run_bit_identical():
    """The bench's headline launches (decode_attention_plan, whose planner also
    describes every attention CTA's first segment, then decode_attention_run) give
    the same bits as decode_attention, whose CTAs work their first segment out
    themselves, on the full-size mixed batch; the latter is checked against the
    oracle on every row above."""
    batch = make_decode_batch(MIXED, device="cuda")
    q, k, v = batch.q, batch.k_pages, batch.v_pages
    bt = torch.from_numpy(batch.block_table).cuda()
    cl = torch.from_numpy(batch.context_lens).cuda()
    out, lse = cadkv.decode_attention(q, k, v, bt, cl)
    out2, lse2 = torch.empty_like(out), torch.empty_like(lse)
    ws = torch.empty(cadkv.decode_attention_workspace_size(MIXED.batch, 64, 8, 128, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    cadkv.decode_attention_plan(q, k, v, bt, cl, out2, lse2, ws)
    cadkv.decode_attention_run(q, k, v, bt, cl, out2, lse2, ws)
    torch.cuda.synchronize()
    assert cadkv.decode_attention_status(ws) == 0
    assert torch.equal(out, out2) and torch.equal(lse, lse2)
    del batch, q, k, v
    torch.cuda.empty_cache()


@pytest.mark.parametrize("slice_pages", [61, 4096, 1 << 20])
def test_mixed_full_size_forced_slices_every_row(slice_pages):
    """The full-size mixed batch with the work slices forced short (many
    partials per trajectory-head), at the planner's dynamic-slice length and
    unsplit: every row against the oracle."""
    batch = make_decode_batch(MIXED, device="cuda")
    tensors = (batch.q, batch.k_pages, batch.v_pages,
               torch.from_numpy(batch.block_table).cuda(),
               torch.from_numpy(batch.context_lens).cuda())
    out, lse = gpu_decode(batch, slice_pages=slice_pages, tensors=tensors)
    ref, ref_lse = full_oracle(batch)
    assert_close(out, lse, ref, ref_lse, f"mixed, slice_pages={slice_pages}")
    del batch, tensors
    torch.cuda.empty_cache()


@pytest.mark.parametrize("slice_pages", [0, 3])
def test_large_batch_every_row(slice_pages):
    """6,000 trajectories (above the batch size up to which a 256-thread planner
    runs and describes the CTAs' first segments: here the 1,024-thread planner
    scans the lengths in six rounds), lengths U[0, 600] with some empty, 8/2
    heads, D = 64; automatic and forced short slices; every row against the
    oracle, through the planner and attention launches separately as well."""
    rng = np.random.Generator(np.random.PCG64(660))
    lens = rng.integers(0, 601, 6000).astype(np.int32)
    lens[::97] = 0
    batch = make_batch(lens, 8, 2, 64, seed=661)
    q, k, v, bt, cl = device_tensors(batch)
    out, lse = gpu_decode(batch, slice_pages=slice_pages, tensors=(q, k, v, bt, cl))
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, f"B=6000, slice_pages={slice_pages}")
    out2, lse2 = torch.empty_like(out), torch.empty_like(lse)
    ws = torch.empty(cadkv.decode_attention_workspace_size(6000, 8, 2, 64, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    cadkv.decode_attention_plan(q, k, v, bt, cl, out2, lse2, ws, slice_pages=slice_pages)
    cadkv.decode_attention_run(q, k, v, bt, cl, out2, lse2, ws)
    torch.cuda.synchronize()
    assert torch.equal(out, out2) and torch.equal(lse, lse2)


@pytest.mark.parametrize("slice_pages", [0, 5])
@pytest.mark.parametrize("hq,hkv,d", [(16, 2, 64), (40, 8, 128)], ids=["G8-D64", "G5-D128"])
def test_mid_size_heavy_tailed_every_row(hq, hkv, d, slice_pages):
    """A mid-size heavy-tailed batch, 300 trajectories with lengths lognormal
    (median 600) clipped to [1, 20,000], for head_dim 64 (the 32-stage ring of
    4 KB stages) and for Qwen3-14B's 40/8 heads (G = 5, three padded query rows
    per MMA tile); automatic slicing and forced short slices (dynamic, many
    partials); every row against the oracle."""
    rng = np.random.Generator(np.random.PCG64(640))
    lens = np.clip(np.round(600 * np.exp(rng.normal(0, 1.2, 300))), 1, 20000).astype(np.int32)
    batch = make_batch(lens, hq, hkv, d, seed=641 + d)
    out, lse = gpu_decode(batch, slice_pages=slice_pages)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, f"{hq}/{hkv} heads D={d}, slice_pages={slice_pages}")


@pytest.mark.parametrize("g,d", [(1, 64), (2, 128), (4, 64), (8, 128), (8, 64), (3, 128),
                                 (5, 128)])
def test_edge_lengths(g, d):
    lens = [0, 1, 2, 15, 16, 17, 31, 32, 33, 255, 256, 257, 1000]
    hkv = 2
    batch = make_batch(lens, g * hkv, hkv, d, seed=100 + g * 10 + d)
    out, lse = gpu_decode(batch)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, f"G={g} D={d}")
    assert torch.all(out[0] == 0)
    assert torch.all(torch.isneginf(lse[0]))


def test_all_trajectories_empty():
    batch = make_batch([0, 0, 0], 8, 2, 128, seed=3)
    out, lse = gpu_decode(batch)
    assert torch.all(out == 0)
    assert torch.all(torch.isneginf(lse))


def test_single_long_trajectory_at_table_limit():
    max_pages = 512
    batch = make_batch([max_pages * 16], 8, 1, 128, seed=4, max_pages=max_pages)
    out, lse = gpu_decode(batch)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, "n = 16 * max_pages")


@pytest.mark.parametrize("slice_pages", [1, 2, 3, 7, 16, 64, 1000, 1 << 20])
def test_split_count_invariance(slice_pages):
    """Forcing the work-slice length (how many partials each trajectory-head is
    split into, and where) stays within tolerance of the oracle."""
    batch = make_batch([3, 40, 700, 1900, 17, 5000], 16, 2, 128, seed=5)
    out, lse = gpu_decode(batch, slice_pages=slice_pages)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, f"slice_pages={slice_pages}")


def test_page_permutation_is_bit_identical():
    """Moving physical pages (same logical content) changes no output bit: the
    work split depends only on lengths."""
    batch = make_batch([100, 513, 37, 2048], 16, 2, 128, seed=6, extra_pages=9)
    out1, lse1 = gpu_decode(batch)
    rng = np.random.Generator(np.random.PCG64(60))
    perm = rng.permutation(batch.num_pages)          # new physical index of page p
    inv = np.argsort(perm)
    k2 = batch.k_pages[torch.from_numpy(inv)]
    v2 = batch.v_pages[torch.from_numpy(inv)]
    table2 = np.where(batch.block_table >= 0, perm[np.maximum(batch.block_table, 0)], -1)
    b2 = DecodeBatch(batch.workload, batch.context_lens, table2.astype(np.int32), batch.q,
                     k2, v2)
    out2, lse2 = gpu_decode(b2)
    assert torch.equal(out1, out2)
    assert torch.equal(lse1, lse2)


def test_deterministic_across_calls():
    batch = make_batch([4000, 9000, 123, 77777 // 16], 32, 8, 128, seed=7)
    tensors = device_tensors(batch)
    a = gpu_decode(batch, tensors=tensors)
    b = gpu_decode(batch, tensors=tensors)
    assert torch.equal(a[0], b[0]) and torch.equal(a[1], b[1])


def test_batch_order_invariance():
    batch = make_batch([5, 900, 60, 3000, 1], 8, 2, 64, seed=8)
    out, lse = gpu_decode(batch)
    order = np.array([3, 0, 4, 1, 2])
    b2 = DecodeBatch(batch.workload, batch.context_lens[order], batch.block_table[order],
                     batch.q[torch.from_numpy(order)], batch.k_pages, batch.v_pages)
    out2, lse2 = gpu_decode(b2)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out2, lse2, ref[order], ref_lse[order], "permuted batch")
    assert_close(out[torch.from_numpy(order).cuda()], lse[torch.from_numpy(order).cuda()],
                 ref[order], ref_lse[order], "original batch")


def test_gqa_matches_replicated_mha():
    batch = make_batch([300, 45], 8, 2, 128, seed=9, nan_tails=False)
    out, lse = gpu_decode(batch)
    k_r = batch.k_pages.repeat_interleave(4, dim=1)
    v_r = batch.v_pages.repeat_interleave(4, dim=1)
    mha = DecodeBatch(batch.workload, batch.context_lens, batch.block_table, batch.q, k_r, v_r)
    out2, lse2 = gpu_decode(mha)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, "GQA")
    assert_close(out2, lse2, ref, ref_lse, "replicated MHA")


def test_closed_forms_on_gpu():
    """q = 0 gives mean V and lse = ln n; n = 1 returns V exactly."""
    batch = make_batch([1, 50, 333], 8, 2, 128, seed=10)
    batch.q.zero_()
    batch.q[0].normal_()          # trajectory 0 (n = 1) keeps a random query
    out, lse = gpu_decode(batch)
    v = batch.v_pages.float()
    for b, n in enumerate(batch.context_lens):
        rows = [v[batch.block_table[b, t // 16], :, t % 16, :] for t in range(int(n))]
        vs = torch.stack(rows)                       # [n, Hkv, D]
        for h in range(8):
            if b == 0:
                assert torch.equal(out[0, h].cpu(), batch.v_pages[batch.block_table[0, 0], h // 4, 0])
            else:
                mean = vs[:, h // 4].double().mean(0).numpy()
                err = np.abs(out[b, h].float().cpu().numpy() - mean).max()
                assert err <= 1e-2, err
                assert abs(lse[b, h].item() - np.log(n)) <= 1e-3 * np.log(n)


def test_lse_is_optional():
    batch = make_batch([70, 5], 4, 1, 64, seed=11)
    out1, _ = gpu_decode(batch)
    out2, lse2 = gpu_decode(batch, want_lse=False)
    assert lse2 is None
    assert torch.equal(out1, out2)


def test_plan_then_run_equals_single_call():
    batch = make_batch([700, 12, 3300], 16, 2, 128, seed=12)
    q, k, v, bt, cl = device_tensors(batch)
    out, lse = cadkv.decode_attention(q, k, v, bt, cl)
    out2 = torch.empty_like(out)
    lse2 = torch.empty_like(lse)
    ws = torch.empty(cadkv.decode_attention_workspace_size(3, 16, 2, 128, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    cadkv.decode_attention_plan(q, k, v, bt, cl, out2, lse2, ws)
    cadkv.decode_attention_run(q, k, v, bt, cl, out2, lse2, ws)
    torch.cuda.synchronize()
    assert torch.equal(out, out2) and torch.equal(lse, lse2)
    assert cadkv.decode_attention_status(ws) == 0


def test_decode_step_matches_decode_attention():
    """The binding's prepared call over fixed buffers gives decode_attention's
    bits, call after call, as the inputs change in place."""
    batch = make_batch([700, 12, 3300, 1], 16, 2, 128, seed=16)
    q, k, v, bt, cl = device_tensors(batch)
    out = torch.empty_like(q)
    lse = torch.empty((4, 16), dtype=torch.float32, device="cuda")
    ws = torch.empty(cadkv.decode_attention_workspace_size(4, 16, 2, 128, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    step = cadkv.DecodeStep(q, k, v, bt, cl, out, lse, ws)
    for i in range(2):
        if i:
            q.mul_(-0.5)                      # new values in the same buffers
        ref_out, ref_lse = cadkv.decode_attention(q, k, v, bt, cl)
        step()
        torch.cuda.synchronize()
        assert torch.equal(out, ref_out) and torch.equal(lse, ref_lse)
    # one prepared plan, then prepared runs over two layers' pages
    k2, v2 = torch.flip(k, dims=[0]), torch.flip(v, dims=[0])
    bt2 = (k.shape[0] - 1 - bt).where(bt >= 0, bt)   # the same logical pages, moved
    plan = cadkv.DecodeStep(q, k, v, bt, cl, out, lse, ws, launch="plan")
    runs = [cadkv.DecodeStep(q, k, v, bt, cl, out, lse, ws, launch="run"),
            cadkv.DecodeStep(q, k2, v2, bt2, cl, out, lse, ws, launch="run")]
    ref_out, ref_lse = cadkv.decode_attention(q, k, v, bt, cl)
    plan()
    for run in runs + runs:
        out.fill_(float("nan"))
        run()
        torch.cuda.synchronize()
        assert torch.equal(out, ref_out) and torch.equal(lse, ref_lse)


@pytest.mark.parametrize("slice_pages", [0, 7, 3, 1])
def test_plan_once_run_per_layer(slice_pages):
    """One plan, then one run per layer (other q, pages and outputs, same
    lengths), twice over: every run matches the oracle, including the rows of
    an empty trajectory, which the planner never wrote for layers 1 and 2.
    The batch has 766 page-heads: slice_pages = 3 and 1 cut 256 and 608 slices,
    more than the CTAs, so every run hands slices out through the counter the
    previous run put back, and merges many partials through arrival counters
    the previous run cleared."""
    lens = [700, 0, 3300, 1, 45, 2048]
    hq, hkv, d = 16, 2, 128
    layers = [make_batch(lens, hq, hkv, d, seed=170 + l) for l in range(3)]  # own tables
    cl = torch.from_numpy(layers[0].context_lens).cuda()
    qs, ks, vs, bts, outs, lses, refs = [], [], [], [], [], [], []
    for b in layers:
        qs.append(b.q.cuda())
        ks.append(b.k_pages.cuda())
        vs.append(b.v_pages.cuda())
        bts.append(torch.from_numpy(b.block_table).cuda())
        outs.append(torch.full_like(qs[-1], float("nan")))
        lses.append(torch.full((len(lens), hq), float("nan"), device="cuda"))
        refs.append(oracle_decode(b))
    width = bts[0].shape[1]
    assert all(t.shape[1] == width for t in bts)
    ws = torch.empty(cadkv.decode_attention_workspace_size(len(lens), hq, hkv, d, width),
                     dtype=torch.uint8, device="cuda")
    cadkv.decode_attention_plan(qs[0], ks[0], vs[0], bts[0], cl, outs[0], lses[0], ws,
                                slice_pages=slice_pages)
    for pass_ in range(2):
        for l in range(3):
            if pass_:
                outs[l].fill_(float("nan"))
                lses[l].fill_(float("nan"))
            cadkv.decode_attention_run(qs[l], ks[l], vs[l], bts[l], cl, outs[l], lses[l], ws)
        torch.cuda.synchronize()
        assert cadkv.decode_attention_status(ws) == 0
        for l in range(3):
            assert_close(outs[l], lses[l], refs[l][0], refs[l][1], f"pass {pass_} layer {l}")
            assert torch.all(outs[l][1] == 0) and torch.all(torch.isneginf(lses[l][1]))


def test_status_reports_bad_page_without_faulting():
    batch = make_batch([40, 20], 4, 1, 64, seed=13, nan_tails=False)
    q, k, v, bt, cl = device_tensors(batch)
    bt[1, 0] = batch.num_pages + 5                   # outside the pool
    ws = torch.empty(cadkv.decode_attention_workspace_size(2, 4, 1, 64, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    out, lse = cadkv.decode_attention(q, k, v, bt, cl, workspace=ws)
    assert cadkv.decode_attention_status(ws) == STATUS["CADKV_ERR_OOB"]
    ref, ref_lse = oracle_decode(DecodeBatch(batch.workload, batch.context_lens[:1],
                                             batch.block_table[:1], batch.q[:1],
                                             batch.k_pages, batch.v_pages))
    assert_close(out[:1], lse[:1], ref, ref_lse, "untouched trajectory")
    # the next good call clears the status
    bt[1, 0] = int(batch.block_table[1, 0])
    cadkv.decode_attention(q, k, v, bt, cl, workspace=ws)
    assert cadkv.decode_attention_status(ws) == 0


def test_status_reports_length_beyond_table():
    batch = make_batch([40, 20], 4, 1, 64, seed=14, nan_tails=False)
    q, k, v, bt, cl = device_tensors(batch)
    cl[1] = bt.shape[1] * 16 + 1
    ws = torch.empty(cadkv.decode_attention_workspace_size(2, 4, 1, 64, bt.shape[1]),
                     dtype=torch.uint8, device="cuda")
    out, lse = cadkv.decode_attention(q, k, v, bt, cl, workspace=ws)
    assert cadkv.decode_attention_status(ws) == STATUS["CADKV_ERR_SHAPE"]
    assert torch.all(out[1] == 0) and torch.all(torch.isneginf(lse[1]))


def test_workspace_too_small_is_rejected():
    batch = make_batch([40], 4, 1, 64, seed=15)
    q, k, v, bt, cl = device_tensors(batch)
    ws = torch.empty(64, dtype=torch.uint8, device="cuda")
    with pytest.raises(cadkv.CadkvError) as e:
        cadkv.decode_attention(q, k, v, bt, cl, workspace=ws)
    assert e.value.status == STATUS["CADKV_ERR_WORKSPACE"]


@pytest.mark.parametrize("b,c", [(32, 16384), (8, 65536), (512, 1024), (512, 256),
                                 (2048, 256)])
def test_landscape_cells_every_row(b, c):
    """Cells of the (B, mean context) landscape sweep at full size, every row
    against the oracle (the two cells of mean 256 take the per-warp mode)."""
    from paper_2609_36899_gb300.workloads import landscape_workload
    w = landscape_workload(b, c)
    batch = make_decode_batch(w, device="cuda")
    tensors = (batch.q, batch.k_pages, batch.v_pages,
               torch.from_numpy(batch.block_table).cuda(),
               torch.from_numpy(batch.context_lens).cuda())
    out, lse = gpu_decode(batch, tensors=tensors)
    ref, ref_lse = full_oracle(batch)
    assert_close(out, lse, ref, ref_lse, w.name)
    del batch, tensors
    torch.cuda.empty_cache()


@pytest.mark.parametrize("comp", ["equal", "lognormal", "bimodal", "one_giant"])
def test_composition_cells_every_row(comp):
    """The within-batch composition sweep at B = 128, mean 4096 (full size as
    benched; one_giant gives one trajectory half of all tokens), every row
    against the oracle."""
    from paper_2609_36899_gb300.workloads import composition_workload
    w = composition_workload(128, 4096, comp)
    batch = make_decode_batch(w, device="cuda")
    tensors = (batch.q, batch.k_pages, batch.v_pages,
               torch.from_numpy(batch.block_table).cuda(),
               torch.from_numpy(batch.context_lens).cuda())
    out, lse = gpu_decode(batch, tensors=tensors)
    ref, ref_lse = full_oracle(batch)
    assert_close(out, lse, ref, ref_lse, w.name)
    del batch, tensors
    torch.cuda.empty_cache()


def test_hbm_read_probe_reads_every_word():
    g = torch.Generator().manual_seed(1)
    host = torch.randint(-2**31, 2**31 - 1, (1 << 20,), generator=g, dtype=torch.int64)
    host = host.to(torch.int32)
    buf = host.cuda()
    sink = torch.zeros(1, dtype=torch.int64, device="cuda")
    cadkv.cadkv_hbm_read_probe(buf, sink)
    torch.cuda.synchronize()
    expect = int(np.bitwise_xor.reduce(host.numpy().view(np.uint32)))
    assert int(sink.item()) & 0xFFFFFFFF == expect
    assert int(sink.item()) >> 32 == 0


def test_bounded_wait_gives_up_and_context_stays_usable():
    """The failure path, run on purpose: a kernel holding tensor memory waits with
    the library's bounded wait on a barrier phase nothing completes.  It must give
    up after the limit, report CADKV_ERR_TIMEOUT in the status word, free its
    resources and leave the context usable for the next call."""
    import time
    ws = torch.zeros(4096, dtype=torch.uint8, device="cuda")
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    cadkv.cadkv_wait_selftest(50_000_000, ws)            # 50 ms
    assert cadkv.kv_prefix_stage_status(ws) == STATUS["CADKV_ERR_TIMEOUT"]
    assert time.perf_counter() - t0 >= 0.045
    batch = make_batch([5, 100, 1000], 8, 2, 128, seed=77)  # the next call still works
    out, lse = gpu_decode(batch)
    ref, ref_lse = oracle_decode(batch)
    assert_close(out, lse, ref, ref_lse, "decode after the self-test")
