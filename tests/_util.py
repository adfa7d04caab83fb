"""Test helpers: bf16 bit conversions and small hand-built paged batches.

These helpers only move data around (rounding to bf16, building block tables);
none of the attention or staging arithmetic lives here.
"""
import numpy as np
import torch


def to_bf16_bits(x) -> np.ndarray:
    """Round float values to bf16 (round-to-nearest-even) and return the bits."""
    t = torch.as_tensor(np.asarray(x, dtype=np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16).copy()


def bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact widening of bf16 bit patterns to float64."""
    u = bits.astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def exact_bf16(x) -> np.ndarray:
    """Assert that x is exactly representable in bf16 and return its bits."""
    bits = to_bf16_bits(x)
    back = bits_to_f64(bits)
    assert np.array_equal(back, np.asarray(x, dtype=np.float64)), "not bf16-exact"
    return bits


def paged(tokens, page_size: int, perm=None, num_pages: int | None = None,
          fill=0):
    """Lay out per-trajectory token rows (a list of [n_b][Hkv][D] arrays) in a
    paged pool [num_pages][Hkv][P][D] of the same dtype: the j-th page of
    trajectory b goes to physical page perm[pos] where pos counts pages of
    trajectories 0..b in order.  Slots and pages not written hold ``fill``.

    Returns (pool, block_table int32 [B, max_pages] with -1 past the end,
    context_lens int32 [B]).
    """
    lens = np.array([t.shape[0] for t in tokens], dtype=np.int32)
    hkv, d = tokens[0].shape[1], tokens[0].shape[2]
    pages = [-(-int(n) // page_size) for n in lens]
    used = sum(pages)
    if num_pages is None:
        num_pages = max(used, 1)
    if perm is None:
        perm = np.arange(num_pages)
    pool = np.full((num_pages, hkv, page_size, d), fill, dtype=tokens[0].dtype)
    max_pages = max(max(pages), 1)
    table = np.full((len(tokens), max_pages), -1, dtype=np.int32)
    pos = 0
    for b, (rows, p) in enumerate(zip(tokens, pages)):
        for j in range(p):
            phys = int(perm[pos])
            pos += 1
            table[b, j] = phys
            chunk = rows[j * page_size:(j + 1) * page_size]
            pool[phys, :, :chunk.shape[0], :] = np.transpose(chunk, (1, 0, 2))
    return pool, table, lens
