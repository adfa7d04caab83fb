"""Helpers for the GPU parity tests: run the CUDA path through the binding and
the oracle on the same bf16 bits, and compare within the stated tolerances.

Tolerances (decode attention): max |out_gpu - out_oracle| <= 1e-2 and
|lse_gpu - lse_oracle| <= 1e-3 * max(|lse_oracle|, 1): relative, with a floor
of 1 where the reference lse itself comes near zero (a trajectory of one or a
few tokens whose scores are near zero; there the relative error of even a
correctly rounded result is unbounded).  Prefix staging: bit-exact.
"""
import numpy as np
import torch

import oracle
import paper_2609_36899_gb300 as cadkv
from paper_2609_36899_gb300.workloads import (DecodeBatch, DecodeWorkload, bf16_bits,
                                              scatter_block_table)

OUT_ATOL = 1e-2
LSE_RTOL = 1e-3
NAN_BF16 = 0x7FC1


def device_tensors(batch: DecodeBatch, device="cuda"):
    q = batch.q.to(device)
    k = batch.k_pages.to(device)
    v = batch.v_pages.to(device)
    bt = torch.from_numpy(batch.block_table).to(device)
    cl = torch.from_numpy(batch.context_lens).to(device)
    return q, k, v, bt, cl


def gpu_decode(batch: DecodeBatch, slice_pages=0, want_lse=True, tensors=None):
    q, k, v, bt, cl = tensors if tensors is not None else device_tensors(batch)
    out, lse = cadkv.decode_attention(q, k, v, bt, cl, slice_pages=slice_pages,
                                      want_lse=want_lse)
    torch.cuda.synchronize()
    return out, lse


def oracle_decode(batch: DecodeBatch, rows=None):
    return oracle.decode_attention(bf16_bits(batch.q), bf16_bits(batch.k_pages),
                                   bf16_bits(batch.v_pages), batch.block_table,
                                   batch.context_lens, rows=rows)


def assert_close(out_gpu, lse_gpu, out_ref, lse_ref, what=""):
    """out_gpu: bf16 tensor; lse_gpu: fp32 tensor or None; refs: float64 numpy."""
    o = out_gpu.float().cpu().numpy().astype(np.float64).reshape(out_ref.shape)
    assert np.all(np.isfinite(o)), f"{what}: non-finite output"
    err = np.abs(o - out_ref).max(initial=0.0)
    assert err <= OUT_ATOL, f"{what}: max |out err| = {err:.3e} > {OUT_ATOL}"
    if lse_gpu is not None:
        _assert_lse(lse_gpu, lse_ref, what)
    return err


def _assert_lse(lse_gpu, lse_ref, what):
    l = lse_gpu.cpu().numpy().astype(np.float64).reshape(lse_ref.shape)
    inf_ref = np.isneginf(lse_ref)
    assert np.array_equal(np.isneginf(l), inf_ref), f"{what}: -inf lse mismatch"
    fin = ~inf_ref
    if fin.any():
        rel = np.abs(l[fin] - lse_ref[fin]) / np.maximum(np.abs(lse_ref[fin]), 1.0)
        assert rel.max() <= LSE_RTOL, f"{what}: max lse rel err = {rel.max():.3e}"


U_BF16 = 2.0 ** -8   # unit roundoff of bf16 (8-bit significand)


def abs_bits(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns with the sign bit cleared: |x| (NaN stays NaN)."""
    return bits & np.uint16(0x7FFF)


def assert_close_bounded(out_gpu, lse_gpu, out_ref, lse_ref, absv_ref, what=""):
    """assert_close with each output element's bound raised to what the
    arithmetic itself guarantees, where that is larger than 1e-2.

    Both kernels round the softmax weights P to bf16 before the P.V product
    (tensor-core operands have one type, and V is bf16) and round out to bf16;
    the row sum comes from the unrounded P.  With u = 2^-8 and w_j the exact
    weights, out_gpu = (1 + e)(sum_j w_j (1 + d_j) v_j) with |d_j|, |e| <= u, so
    |out_gpu - out_ref| <= u (sum_j w_j |v_j| + |out_ref|) up to fp32 rounding.
    `absv_ref` is sum_j w_j |v_j| per element: the oracle run on |V|.  Rows over
    many keys stay at 1e-2 (the bound is ~3e-3 there); a row over a handful of
    keys whose values are large (|v| ~ 4) can reach ~1.5e-2, and gets the bound.
    """
    o = out_gpu.float().cpu().numpy().astype(np.float64).reshape(out_ref.shape)
    assert np.all(np.isfinite(o)), f"{what}: non-finite output"
    bound = U_BF16 * (absv_ref + np.abs(out_ref)) * 1.01 + 1e-4
    tol = np.maximum(OUT_ATOL, bound)
    excess = np.abs(o - out_ref) - tol
    worst = np.unravel_index(np.argmax(excess), excess.shape)
    assert excess[worst] <= 0, (f"{what}: |out err| {abs(o - out_ref)[worst]:.3e} > "
                                f"bound {tol[worst]:.3e} at {tuple(int(i) for i in worst)}")
    if lse_gpu is not None:
        _assert_lse(lse_gpu, lse_ref, what)


def make_batch(lens, hq, hkv, d, seed, extra_pages=5, max_pages=None, nan_tails=True,
               k_scale=1.0):
    """A decode batch with the given context lengths on the CPU.

    Pages are a seeded permutation of the pool; slots past n_b, unused pages and
    table entries past the last page hold NaN / -1 when ``nan_tails``.
    """
    lens = np.asarray(lens, dtype=np.int32)
    pages = -(-lens.astype(np.int64) // 16)
    if max_pages is None:
        max_pages = max(int(pages.max(initial=0)), 1)
    rng = np.random.Generator(np.random.PCG64(seed))
    used = int(pages.sum())
    table, pool_pages = scatter_block_table(lens, 16, max_pages, used + extra_pages, rng)
    gen = torch.Generator().manual_seed(seed)
    q = torch.randn((len(lens), hq, d), generator=gen).to(torch.bfloat16)
    k = (torch.randn((pool_pages, hkv, 16, d), generator=gen) * k_scale).to(torch.bfloat16)
    v = torch.randn((pool_pages, hkv, 16, d), generator=gen).to(torch.bfloat16)
    if nan_tails:
        used_mask = np.zeros((pool_pages, 16), dtype=bool)
        for b, n in enumerate(lens):
            for j in range(int(pages[b])):
                cnt = min(16, int(n) - 16 * j)
                used_mask[table[b, j], :cnt] = True
        m = torch.from_numpy(~used_mask)
        for t in (k, v):
            tv = t.view(torch.int16)
            tv[m[:, None, :, None].expand_as(tv)] = NAN_BF16
    w = DecodeWorkload("custom", len(lens), hq, hkv, d, "fixed", tuple(int(x) for x in lens),
                       16 * max_pages, seed)
    return DecodeBatch(w, lens, table, q, k, v)


def sampled_oracle(batch_dev: DecodeBatch, sample_b):
    """Oracle for a few trajectories of a device-resident batch: copy only their
    pages to the host and renumber them 0..p-1 (page placement does not change
    the result -- pinned by the oracle's page-permutation pin)."""
    lens = batch_dev.context_lens[sample_b]
    pages = -(-lens.astype(np.int64) // 16)
    max_p = max(int(pages.max(initial=1)), 1)
    phys = np.concatenate([batch_dev.block_table[b, :p] for b, p in zip(sample_b, pages)])
    idx = torch.from_numpy(phys.astype(np.int64)).to(batch_dev.k_pages.device)
    k = bf16_bits(batch_dev.k_pages.index_select(0, idx)) if len(phys) else None
    v = bf16_bits(batch_dev.v_pages.index_select(0, idx)) if len(phys) else None
    table = np.full((len(sample_b), max_p), -1, dtype=np.int32)
    pos = 0
    for i, p in enumerate(pages):
        table[i, :p] = np.arange(pos, pos + p)
        pos += p
    q = bf16_bits(batch_dev.q[torch.as_tensor(np.asarray(sample_b), device=batch_dev.q.device)])
    return oracle.decode_attention(q, k, v, table, lens)


def full_oracle(batch_dev: DecodeBatch, max_group_bytes=2 << 30):
    """Oracle for EVERY trajectory of a device-resident batch.

    Trajectories are taken in order, in groups whose K and V pages fit in
    ``max_group_bytes`` of host memory; each group goes through
    ``sampled_oracle``.  Returns (out float64 [B, Hq, D], lse float64 [B, Hq]).
    """
    lens = batch_dev.context_lens
    _, hkv, page, d = batch_dev.k_pages.shape
    page_bytes = 2 * hkv * page * d * 2
    pages = -(-lens.astype(np.int64) // 16)
    outs, lses, group, acc = [], [], [], 0
    for b in range(len(lens)):
        need = int(pages[b]) * page_bytes
        if group and acc + need > max_group_bytes:
            o, l = sampled_oracle(batch_dev, group)
            outs.append(o)
            lses.append(l)
            group, acc = [], 0
        group.append(b)
        acc += need
    if group:
        o, l = sampled_oracle(batch_dev, group)
        outs.append(o)
        lses.append(l)
    return np.concatenate(outs), np.concatenate(lses)
