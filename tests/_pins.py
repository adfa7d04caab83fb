"""Pins for the fp64 oracle: checks against facts that do not come from the
oracle itself -- library routines on special cases, closed forms, invariants
and a hand-worked example.

Each pin is a function ``pin_*(orc)`` that raises AssertionError when the
oracle ``orc`` (an ``oracle.Oracle``) disagrees.  ``test_oracle_attention.py``
and ``test_oracle_staging.py`` run them against the real oracle;
``test_oracle_mutants.py`` runs them against deliberately broken copies of
``oracle.c`` and requires every mutant to fail at least one pin.
"""
import json
import math
import os

import numpy as np
import scipy.special as sp

from _util import bits_to_f64, exact_bf16, paged, to_bf16_bits

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")
NAN_BF16 = np.uint16(0x7FC1)


def _rng(seed):
    return np.random.Generator(np.random.PCG64(seed))


def _random_batch(seed, lens, hq, hkv, d, page_size=16, extra_pages=3, scale=1.0):
    """Random bf16 batch with a shuffled pool; returns logical rows too."""
    rng = _rng(seed)
    q = to_bf16_bits(rng.normal(size=(len(lens), hq, d)))
    ks = [to_bf16_bits(scale * rng.normal(size=(n, hkv, d))) for n in lens]
    vs = [to_bf16_bits(rng.normal(size=(n, hkv, d))) for n in lens]
    used = sum(-(-n // page_size) for n in lens)
    num_pages = used + extra_pages
    perm = rng.permutation(num_pages)
    kp, table, cl = paged(ks, page_size, perm, num_pages)
    vp, _, _ = paged(vs, page_size, perm, num_pages)
    return q, kp, vp, table, cl, ks, vs


def _scipy_reference(q, ks, vs, hq, hkv):
    """softmax(q K^T / sqrt(D)) V per (b, h) with scipy, from logical rows."""
    b_n, _, d = q.shape
    g = hq // hkv
    out = np.zeros((b_n, hq, d))
    lse = np.full((b_n, hq), -np.inf)
    for b in range(b_n):
        if ks[b].shape[0] == 0:
            continue
        for h in range(hq):
            kf = bits_to_f64(ks[b][:, h // g, :])
            vf = bits_to_f64(vs[b][:, h // g, :])
            s = kf @ bits_to_f64(q[b, h]) / math.sqrt(d)
            out[b, h] = sp.softmax(s) @ vf
            lse[b, h] = sp.logsumexp(s)
    return out, lse


# --------------------------------------------------------------------------
# decode attention
# --------------------------------------------------------------------------

def pin_attention_matches_scipy_mha(orc):
    """One head, one trajectory, ragged last page: scipy softmax/logsumexp."""
    q, kp, vp, table, cl, ks, vs = _random_batch(1, [50], 1, 1, 64)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    ref, ref_lse = _scipy_reference(q, ks, vs, 1, 1)
    np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-12, atol=1e-12)


def pin_attention_matches_scipy_gqa_paged(orc):
    """GQA (G = 4), several trajectories, shuffled pages, ragged tails."""
    lens = [17, 64, 1, 250, 33]
    q, kp, vp, table, cl, ks, vs = _random_batch(2, lens, 8, 2, 64)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    ref, ref_lse = _scipy_reference(q, ks, vs, 8, 2)
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-12, atol=1e-12)


def pin_attention_zero_query(orc):
    """q = 0: every score is 0, so out = mean of V rows and lse = ln n."""
    lens = [1, 17, 300]
    q, kp, vp, table, cl, ks, vs = _random_batch(3, lens, 4, 2, 64)
    q[:] = 0
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    for b, n in enumerate(lens):
        for h in range(4):
            mean_v = bits_to_f64(vs[b][:, h // 2, :]).mean(axis=0)
            np.testing.assert_allclose(out[b, h], mean_v, rtol=1e-13, atol=1e-14)
            assert abs(lse[b, h] - math.log(n)) <= 1e-13 * max(1.0, math.log(n))


def pin_attention_single_token(orc):
    """n = 1: out is that token's V row, lse is its scaled score."""
    q, kp, vp, table, cl, ks, vs = _random_batch(4, [1, 1], 4, 4, 128)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    for b in range(2):
        for h in range(4):
            np.testing.assert_array_equal(out[b, h], bits_to_f64(vs[b][0, h]))
            s0 = float(np.dot(bits_to_f64(q[b, h]), bits_to_f64(ks[b][0, h])))
            assert abs(lse[b, h] - s0 / math.sqrt(128)) <= 1e-13 * max(1, abs(s0))


def pin_attention_identical_keys(orc):
    """All keys equal: uniform weights, out = mean V, lse = s + ln n."""
    rng = _rng(5)
    n, d = 40, 64
    krow = to_bf16_bits(rng.normal(size=(1, d)))
    ks = [np.repeat(krow[None], n, axis=0)]           # [n][1][D]
    vs = [to_bf16_bits(rng.normal(size=(n, 1, d)))]
    q = to_bf16_bits(rng.normal(size=(1, 1, d)))
    kp, table, cl = paged(ks, 16)
    vp, _, _ = paged(vs, 16)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    np.testing.assert_allclose(out[0, 0], bits_to_f64(vs[0][:, 0]).mean(axis=0),
                               rtol=1e-13, atol=1e-14)
    s = float(np.dot(bits_to_f64(q[0, 0]), bits_to_f64(krow[0]))) / math.sqrt(d)
    assert abs(lse[0, 0] - (s + math.log(n))) <= 1e-12


def pin_attention_dominant_key(orc):
    """One key scores 32 above the rest: out is its V row to ~1e-12."""
    d, n, star = 64, 37, 21
    q = exact_bf16(np.eye(1, d)[None] * 4.0)            # q = 4 e_0
    k = np.zeros((n, 1, d))
    k[star, 0, 0] = 64.0                                # s = 4*64/8 = 32
    rng = _rng(6)
    vs = [to_bf16_bits(rng.normal(size=(n, 1, d)))]
    kp, table, cl = paged([exact_bf16(k)], 16)
    vp, _, _ = paged(vs, 16)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    np.testing.assert_allclose(out[0, 0], bits_to_f64(vs[0][star, 0]), atol=1e-11)
    assert abs(lse[0, 0] - (32.0 + math.log1p((n - 1) * math.exp(-32.0)))) < 1e-12


def pin_attention_page_permutation(orc):
    """Physical page placement does not change the result (same bits)."""
    lens = [40, 7, 129]
    rng = _rng(7)
    q = to_bf16_bits(rng.normal(size=(3, 4, 64)))
    ks = [to_bf16_bits(rng.normal(size=(n, 2, 64))) for n in lens]
    vs = [to_bf16_bits(rng.normal(size=(n, 2, 64))) for n in lens]
    results = []
    for perm_seed, extra in ((0, 0), (1, 5), (2, 11)):
        used = sum(-(-n // 16) for n in lens)
        perm = _rng(100 + perm_seed).permutation(used + extra)
        kp, table, cl = paged(ks, 16, perm, used + extra, fill=NAN_BF16)
        vp, _, _ = paged(vs, 16, perm, used + extra, fill=NAN_BF16)
        results.append(orc.decode_attention(q, kp, vp, table, cl))
    for out, lse in results[1:]:
        np.testing.assert_array_equal(out, results[0][0])
        np.testing.assert_array_equal(lse, results[0][1])


def pin_attention_gqa_equals_replicated_mha(orc):
    """GQA with Hkv heads equals MHA with each KV head repeated G times."""
    lens = [33, 100]
    q, kp, vp, table, cl, ks, vs = _random_batch(8, lens, 8, 2, 64)
    gqa = orc.decode_attention(q, kp, vp, table, cl)
    ks_r = [np.repeat(k, 4, axis=1) for k in ks]        # head h -> kv head h // 4
    vs_r = [np.repeat(v, 4, axis=1) for v in vs]
    kp2, t2, c2 = paged(ks_r, 16)
    vp2, _, _ = paged(vs_r, 16)
    mha = orc.decode_attention(q, kp2, vp2, t2, c2)
    np.testing.assert_array_equal(gqa[0], mha[0])
    np.testing.assert_array_equal(gqa[1], mha[1])


def pin_attention_batch_order(orc):
    """Permuting trajectories permutes the output rows and nothing else."""
    lens = [5, 60, 17, 99]
    q, kp, vp, table, cl, ks, vs = _random_batch(9, lens, 4, 4, 64)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    order = np.array([2, 0, 3, 1])
    out2, lse2 = orc.decode_attention(q[order], kp, vp, table[order], cl[order])
    np.testing.assert_array_equal(out2, out[order])
    np.testing.assert_array_equal(lse2, lse[order])


def pin_attention_key_shift(orc):
    """Adding one vector c to every key adds q.c/sqrt(D) to every score: the
    output is unchanged and lse moves by q.c/sqrt(D).  Small integers keep
    every input exactly representable in bf16."""
    rng = _rng(10)
    n, d = 45, 64
    q = exact_bf16(rng.integers(-2, 3, size=(1, 2, d)).astype(float) / 4)
    k = rng.integers(-4, 5, size=(n, 1, d)).astype(float) / 4
    c = rng.integers(-4, 5, size=(d,)).astype(float) / 4
    vs = [to_bf16_bits(rng.normal(size=(n, 1, d)))]
    vp, table, cl = paged(vs, 16)
    k1, _, _ = paged([exact_bf16(k)], 16)
    k2, _, _ = paged([exact_bf16(k + c)], 16)
    o1, l1 = orc.decode_attention(q, k1, vp, table, cl)
    o2, l2 = orc.decode_attention(q, k2, vp, table, cl)
    np.testing.assert_allclose(o2, o1, rtol=1e-12, atol=1e-13)
    shift = bits_to_f64(q[0]) @ c / math.sqrt(d)
    np.testing.assert_allclose(l2[0], l1[0] + shift, rtol=1e-13, atol=1e-12)


def pin_attention_linear_in_values(orc):
    """The output is linear in V: out(V1 + V2) = out(V1) + out(V2)."""
    rng = _rng(11)
    lens = [29, 64]
    q, kp, _, table, cl, _, _ = _random_batch(11, lens, 4, 2, 64)
    v1 = rng.integers(-8, 9, size=(kp.shape)).astype(float)
    v2 = rng.integers(-8, 9, size=(kp.shape)).astype(float)
    o1, _ = orc.decode_attention(q, kp, exact_bf16(v1), table, cl)
    o2, _ = orc.decode_attention(q, kp, exact_bf16(v2), table, cl)
    o3, _ = orc.decode_attention(q, kp, exact_bf16(v1 + v2), table, cl)
    np.testing.assert_allclose(o3, o1 + o2, rtol=1e-12, atol=1e-12)


def pin_attention_ignores_tail_and_unused(orc):
    """Slots past n_b, unused pages and table entries past the last page never
    reach the result: filling them with NaN instead of 0 changes nothing."""
    lens = [17, 31, 250]
    rng = _rng(12)
    q = to_bf16_bits(rng.normal(size=(3, 4, 64)))
    ks = [to_bf16_bits(rng.normal(size=(n, 2, 64))) for n in lens]
    vs = [to_bf16_bits(rng.normal(size=(n, 2, 64))) for n in lens]
    used = sum(-(-n // 16) for n in lens)
    perm = rng.permutation(used + 4)
    kp, table, cl = paged(ks, 16, perm, used + 4, fill=0)
    vp, _, _ = paged(vs, 16, perm, used + 4, fill=0)
    clean = orc.decode_attention(q, kp, vp, table, cl)
    kp2, _, _ = paged(ks, 16, perm, used + 4, fill=NAN_BF16)
    vp2, _, _ = paged(vs, 16, perm, used + 4, fill=NAN_BF16)
    wide = np.full((table.shape[0], table.shape[1] + 3), -1, dtype=np.int32)
    wide[:, :table.shape[1]] = table
    dirty = orc.decode_attention(q, kp2, vp2, wide, cl)
    np.testing.assert_array_equal(dirty[0], clean[0])
    np.testing.assert_array_equal(dirty[1], clean[1])


def pin_attention_empty_trajectory(orc):
    """n_b = 0 gives out = 0 and lse = -inf; its neighbours are unaffected."""
    lens = [0, 20, 0]
    q, kp, vp, table, cl, ks, vs = _random_batch(13, lens, 2, 1, 64)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    assert np.all(out[0] == 0) and np.all(out[2] == 0)
    assert np.all(np.isneginf(lse[0])) and np.all(np.isneginf(lse[2]))
    ref, ref_lse = _scipy_reference(q, ks, vs, 2, 1)
    np.testing.assert_allclose(out[1], ref[1], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(lse[1], ref_lse[1], rtol=1e-12)


def pin_attention_rows_subset(orc):
    """Evaluating a subset of (b, h) rows gives the same values as the full call."""
    lens = [12, 80, 3]
    q, kp, vp, table, cl, _, _ = _random_batch(14, lens, 4, 2, 64)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    rows = np.array([11, 0, 5, 6])
    o2, l2 = orc.decode_attention(q, kp, vp, table, cl, rows=rows)
    np.testing.assert_array_equal(o2, out.reshape(-1, 64)[rows])
    np.testing.assert_array_equal(l2, lse.reshape(-1)[rows])


def pin_attention_golden_worked_example(orc):
    """Hand-derived example (tests/golden/decode_attention_worked.json)."""
    with open(os.path.join(GOLDEN, "decode_attention_worked.json")) as f:
        g = json.load(f)
    q = exact_bf16(np.array(g["q"], dtype=float))
    kp = exact_bf16(np.array(g["k_pages"], dtype=float))
    vp = exact_bf16(np.array(g["v_pages"], dtype=float))
    mask = np.array(g["nan_mask"], dtype=bool)
    kp[mask] = NAN_BF16
    vp[mask] = NAN_BF16
    table = np.array(g["block_table"], dtype=np.int32)
    cl = np.array(g["context_lens"], dtype=np.int32)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    np.testing.assert_allclose(out, np.array(g["expected_out"]), rtol=0, atol=1e-15)
    np.testing.assert_allclose(lse, np.array(g["expected_lse"]), rtol=0, atol=1e-15)


ATTENTION_PINS = [v for k, v in sorted(globals().items())
                  if k.startswith("pin_attention_")]


# --------------------------------------------------------------------------
# prefix staging and its inverse
# --------------------------------------------------------------------------

def _staging_case(seed, lens, layers, hkv, d, page_size=16, extra=2, perm=True):
    rng = _rng(seed)
    used = sum(-(-n // page_size) for n in lens)
    num_pages = used + extra
    p = rng.permutation(num_pages) if perm else np.arange(num_pages)
    # raw 16-bit patterns, NaN payloads included: staging is a bit copy
    kt = [[rng.integers(0, 1 << 16, size=(n, hkv, d), dtype=np.uint16)
           for n in lens] for _ in range(layers)]
    vt = [[rng.integers(0, 1 << 16, size=(n, hkv, d), dtype=np.uint16)
           for n in lens] for _ in range(layers)]
    kpool = np.stack([paged(kt[l], page_size, p, num_pages, fill=0xFFFF)[0]
                      for l in range(layers)])
    vpool = np.stack([paged(vt[l], page_size, p, num_pages, fill=0xFFFF)[0]
                      for l in range(layers)])
    _, table, cl = paged(kt[0], page_size, p, num_pages)
    return kpool, vpool, table, cl, kt, vt


def pin_stage_brute_force_loop(orc):
    """Element-by-element Python loop over the logical rows."""
    lens = [3, 17, 0, 33]
    L, hkv, d = 3, 2, 8
    kpool, vpool, table, cl, kt, vt = _staging_case(20, lens, L, hkv, d)
    dst = orc.prefix_stage(kpool, vpool, table, cl, 1, 3)
    pos = 0
    for b, n in enumerate(lens):
        for l in (1, 2):
            for kv, src in ((0, kt), (1, vt)):
                for h in range(hkv):
                    for t in range(n):
                        for e in range(d):
                            assert dst[pos] == src[l][b][t, h, e]
                            pos += 1
    assert pos == dst.size


def pin_stage_identity_table_is_slice(orc):
    """With pages laid out in order, each staged row is a reshape of the pool."""
    lens = [20, 48, 5]
    L, hkv, d = 2, 3, 16
    kpool, vpool, table, cl, _, _ = _staging_case(21, lens, L, hkv, d, perm=False)
    dst = orc.prefix_stage(kpool, vpool, table, cl, 0, L)
    pos, first_page = 0, 0
    for b, n in enumerate(lens):
        p = -(-n // 16)
        for l in range(L):
            for pool in (kpool, vpool):
                for h in range(hkv):
                    rows = pool[l, first_page:first_page + p, h].reshape(-1, d)[:n]
                    np.testing.assert_array_equal(dst[pos:pos + n * d], rows.ravel())
                    pos += n * d
        first_page += p


def pin_stage_page_permutation(orc):
    """Staged bytes do not depend on where the pages sit in the pool."""
    lens = [19, 40]
    a = _staging_case(22, lens, 2, 2, 16, perm=True)
    rng = _rng(23)
    used = sum(-(-n // 16) for n in lens)
    p2 = rng.permutation(used + 7)
    k2 = np.stack([paged(a[4][l], 16, p2, used + 7, fill=0)[0] for l in range(2)])
    v2 = np.stack([paged(a[5][l], 16, p2, used + 7, fill=0)[0] for l in range(2)])
    _, t2, c2 = paged(a[4][0], 16, p2, used + 7)
    d1 = orc.prefix_stage(a[0], a[1], a[2], a[3], 0, 2)
    d2 = orc.prefix_stage(k2, v2, t2, c2, 0, 2)
    np.testing.assert_array_equal(d1, d2)


def pin_stage_offsets_and_sentinels(orc):
    """Explicit offsets are honoured and bytes outside the rows are untouched."""
    lens = [9, 16, 1]
    L, hkv, d = 1, 2, 8
    kpool, vpool, table, cl, _, _ = _staging_case(24, lens, L, hkv, d)
    packed = orc.prefix_stage(kpool, vpool, table, cl, 0, L)
    row = L * 2 * hkv * d
    sizes = [n * row for n in lens]
    gap = 5
    offs = np.array([gap, gap + sizes[0] + gap, gap + sizes[0] + gap + sizes[1] + gap])
    total = int(offs[-1] + sizes[-1] + gap)
    dst = np.full(total, 0xABCD, dtype=np.uint16)
    dst = orc.prefix_stage(kpool, vpool, table, cl, 0, L, dst_offsets=offs, dst=dst)
    start = 0
    mask = np.ones(total, dtype=bool)
    for b in range(3):
        np.testing.assert_array_equal(dst[offs[b]:offs[b] + sizes[b]],
                                      packed[start:start + sizes[b]])
        mask[offs[b]:offs[b] + sizes[b]] = False
        start += sizes[b]
    assert np.all(dst[mask] == 0xABCD)


def pin_stage_round_trip(orc):
    """Stage from one pool, load into another with a different table: the new
    pool holds the same logical rows, and restaging gives the same bytes."""
    lens = [21, 64, 2]
    L, hkv, d = 2, 2, 8
    kpool, vpool, table, cl, kt, vt = _staging_case(25, lens, L, hkv, d)
    staged = orc.prefix_stage(kpool, vpool, table, cl, 0, L)
    used = sum(-(-n // 16) for n in lens)
    perm = _rng(26).permutation(used + 3)
    _, t2, _ = paged(kt[0], 16, perm, used + 3)
    k2 = np.zeros((L, used + 3, hkv, 16, d), dtype=np.uint16)
    v2 = np.zeros_like(k2)
    orc.prefix_load(k2, v2, t2, cl, 0, L, staged)
    for l in range(L):
        for b, n in enumerate(lens):
            for t in range(n):
                np.testing.assert_array_equal(k2[l, t2[b, t // 16], :, t % 16], kt[l][b][t])
                np.testing.assert_array_equal(v2[l, t2[b, t // 16], :, t % 16], vt[l][b][t])
    again = orc.prefix_stage(k2, v2, t2, cl, 0, L)
    np.testing.assert_array_equal(again, staged)


STAGE_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_stage_")]


# --------------------------------------------------------------------------
# KV append
# --------------------------------------------------------------------------

def pin_append_then_attend_matches_scipy(orc):
    """Appending the new token's K/V and attending equals scipy attention over
    the logical rows with the new token as the last row."""
    lens_old = [16, 0, 40, 5]
    hq, hkv, d = 8, 2, 64
    rng = _rng(50)
    ks = [to_bf16_bits(rng.normal(size=(n + 1, hkv, d))) for n in lens_old]
    vs = [to_bf16_bits(rng.normal(size=(n + 1, hkv, d))) for n in lens_old]
    q = to_bf16_bits(rng.normal(size=(len(lens_old), hq, d)))
    # pool holds the old rows plus junk in the slot the new token goes to
    junk_k = [np.concatenate([k[:-1], np.full((1, hkv, d), NAN_BF16, np.uint16)]) for k in ks]
    junk_v = [np.concatenate([v[:-1], np.full((1, hkv, d), NAN_BF16, np.uint16)]) for v in vs]
    used = sum(-(-(n + 1) // 16) for n in lens_old)
    perm = rng.permutation(used + 2)
    kp, table, cl = paged(junk_k, 16, perm, used + 2, fill=NAN_BF16)
    vp, _, _ = paged(junk_v, 16, perm, used + 2, fill=NAN_BF16)
    k_new = np.stack([k[-1] for k in ks])
    v_new = np.stack([v[-1] for v in vs])
    orc.kv_append(kp, vp, k_new, v_new, table, cl)
    out, lse = orc.decode_attention(q, kp, vp, table, cl)
    ref, ref_lse = _scipy_reference(q, ks, vs, hq, hkv)
    np.testing.assert_allclose(out, ref, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, rtol=1e-12, atol=1e-12)


def pin_append_writes_only_the_new_slot(orc):
    """Append changes exactly the (page, head, slot) of token n_b - 1 of every
    non-empty trajectory, to the new bits, and nothing else."""
    lens = [1, 16, 17, 0, 33]
    hkv, d = 3, 8
    rng = _rng(51)
    used = sum(-(-n // 16) for n in lens)
    table = np.full((len(lens), 3), -1, dtype=np.int32)
    perm = rng.permutation(used + 2)
    pos = 0
    for b, n in enumerate(lens):
        p = -(-n // 16)
        table[b, :p] = perm[pos:pos + p]
        pos += p
    kp = rng.integers(0, 1 << 16, size=(used + 2, hkv, 16, d), dtype=np.uint16)
    vp = rng.integers(0, 1 << 16, size=(used + 2, hkv, 16, d), dtype=np.uint16)
    k0, v0 = kp.copy(), vp.copy()
    k_new = rng.integers(0, 1 << 16, size=(len(lens), hkv, d), dtype=np.uint16)
    v_new = rng.integers(0, 1 << 16, size=(len(lens), hkv, d), dtype=np.uint16)
    orc.kv_append(kp, vp, k_new, v_new, table, np.array(lens, dtype=np.int32))
    changed = np.zeros(kp.shape[:3], dtype=bool)
    for b, n in enumerate(lens):
        if n == 0:
            continue
        ph, sl = table[b, (n - 1) // 16], (n - 1) % 16
        np.testing.assert_array_equal(kp[ph, :, sl], k_new[b])
        np.testing.assert_array_equal(vp[ph, :, sl], v_new[b])
        changed[ph, :, sl] = True
    np.testing.assert_array_equal(kp[~changed], k0[~changed])
    np.testing.assert_array_equal(vp[~changed], v0[~changed])


APPEND_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_append_")]


# --------------------------------------------------------------------------
# chunked prefill attention
# --------------------------------------------------------------------------

def _prefill_case(seed, lens, chunks, hq, hkv, d):
    rng = _rng(seed)
    ks = [to_bf16_bits(rng.normal(size=(n, hkv, d))) for n in lens]
    vs = [to_bf16_bits(rng.normal(size=(n, hkv, d))) for n in lens]
    used = sum(-(-n // 16) for n in lens)
    perm = rng.permutation(used + 2)
    kp, table, cl = paged(ks, 16, perm, used + 2, fill=NAN_BF16)
    vp, _, _ = paged(vs, 16, perm, used + 2, fill=NAN_BF16)
    offs = np.concatenate([[0], np.cumsum(chunks)]).astype(np.int64)
    q = to_bf16_bits(rng.normal(size=(int(offs[-1]), hq, d)))
    return q, offs, kp, vp, table, cl, ks, vs


def pin_prefill_matches_scipy_causal(orc):
    """Chunk = whole context: causal self-attention, checked row by row with
    scipy softmax over the keys at or before each query's position."""
    lens, chunks = [37, 20], [37, 9]
    hq, hkv, d = 4, 2, 64
    q, offs, kp, vp, table, cl, ks, vs = _prefill_case(60, lens, chunks, hq, hkv, d)
    out, lse = orc.prefill_attention(q, offs, kp, vp, table, cl)
    for b, (n, c) in enumerate(zip(lens, chunks)):
        for i in range(c):
            pos = n - c + i
            row = offs[b] + i
            for h in range(hq):
                kf = bits_to_f64(ks[b][:pos + 1, h // 2])
                vf = bits_to_f64(vs[b][:pos + 1, h // 2])
                s = kf @ bits_to_f64(q[row, h]) / math.sqrt(d)
                np.testing.assert_allclose(out[row, h], sp.softmax(s) @ vf, rtol=1e-11, atol=1e-12)
                assert abs(lse[row, h] - sp.logsumexp(s)) <= 1e-12 * max(1, abs(lse[row, h]))


def pin_prefill_rows_equal_decode_at_their_position(orc):
    """Each prefill row equals decode attention with the trajectory truncated
    to that query's position (same bits)."""
    lens, chunks = [50, 17, 33], [5, 0, 3]
    hq, hkv, d = 8, 2, 64
    q, offs, kp, vp, table, cl, _, _ = _prefill_case(61, lens, chunks, hq, hkv, d)
    out, lse = orc.prefill_attention(q, offs, kp, vp, table, cl)
    rows_b, rows_len = [], []
    for b, (n, c) in enumerate(zip(lens, chunks)):
        for i in range(c):
            rows_b.append(b)
            rows_len.append(n - c + i + 1)
    dec_out, dec_lse = orc.decode_attention(q, kp, vp, table[rows_b],
                                            np.array(rows_len, dtype=np.int32))
    np.testing.assert_array_equal(out, dec_out)
    np.testing.assert_array_equal(lse, dec_lse)


def pin_prefill_is_causal(orc):
    """Changing the last token's K and V changes only the last query row."""
    lens, chunks = [40], [6]
    q, offs, kp, vp, table, cl, ks, vs = _prefill_case(62, lens, chunks, 2, 1, 64)
    a = orc.prefill_attention(q, offs, kp, vp, table, cl)
    t = 39
    ph, sl = table[0, t // 16], t % 16
    kp2, vp2 = kp.copy(), vp.copy()
    kp2[ph, :, sl] = to_bf16_bits(np.full((1, 64), 3.0))
    vp2[ph, :, sl] = to_bf16_bits(np.full((1, 64), -5.0))
    b_ = orc.prefill_attention(q, offs, kp2, vp2, table, cl)
    np.testing.assert_array_equal(a[0][:5], b_[0][:5])
    assert not np.allclose(a[0][5], b_[0][5])


PREFILL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_prefill_")]
