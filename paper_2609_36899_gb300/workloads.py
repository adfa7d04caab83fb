"""Seeded synthetic workloads shaped like rollout decode batches.

This module only draws random inputs: context lengths, block tables and bf16
values.  It holds none of the attention or staging arithmetic, so both the
CUDA path and the CPU oracle can be fed from it without sharing any of the
method's code.

The paper's traces (Qwen3-8B rollouts, Sec. 2.2) are not available; the
length distributions below stand in for their heavy-tailed response lengths,
and values are N(0, 1) bf16 rather than real activations.

Every workload is a pure function of its seed:

* lengths and page permutations come from numpy's PCG64 seeded with ``seed``;
* values come from a ``torch.Generator`` on the target device seeded with
  ``seed`` (for the per-layer staging pool: ``seed * 1000 + layer``).
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

PAGE_SIZE = 16


@dataclass(frozen=True)
class DecodeWorkload:
    """Shape of one decode-attention batch."""
    name: str
    batch: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    lengths: str                     # "fixed" | "uniform" | "lognormal"
    length_args: tuple
    max_len: int                     # block-table width = ceil(max_len / 16)
    seed: int
    pool_pages: int | None = None    # None: exactly the pages the batch uses
    k_scale: float = 1.0
    page_size: int = PAGE_SIZE

    @property
    def max_pages(self) -> int:
        return -(-self.max_len // self.page_size)


@dataclass(frozen=True)
class StagingWorkload:
    """Shape of one late-bound KV prefix-staging job."""
    name: str
    batch: int
    num_layers: int
    num_kv_heads: int
    head_dim: int
    length_args: tuple               # uniform [lo, hi]
    max_len: int
    seed: int
    page_size: int = PAGE_SIZE

    @property
    def max_pages(self) -> int:
        return -(-self.max_len // self.page_size)


TINY = DecodeWorkload("tiny decode attention", 4, 8, 2, 64, "fixed",
                      (17, 64, 250, 1000), 1024, 20261, pool_pages=128)
PACED = DecodeWorkload("paced large batch", 256, 32, 8, 128, "uniform",
                       (1024, 4096), 4096, 20262, k_scale=0.5)
LONG_TAIL = DecodeWorkload("long-context tail", 8, 32, 8, 128, "uniform",
                           (65536, 131072), 131072, 20263)
MIXED = DecodeWorkload("mixed heavy-tailed rollout batch", 512, 64, 8, 128,
                       "lognormal", (4096, 1.0, 512, 131072), 131072, 20264)
STAGING = StagingWorkload("late-bound KV prefix staging", 64, 48, 8, 128,
                          (8192, 65536), 65536, 20265)

DECODE_WORKLOADS = {"tiny": TINY, "paced": PACED, "long_tail": LONG_TAIL,
                    "mixed": MIXED}


@dataclass(frozen=True)
class PrefillWorkload:
    """Shape of one chunked re-prefill job: each of `batch` trajectories of
    `context` tokens recomputes attention for its last `chunk` tokens."""
    name: str
    batch: int
    context: int
    chunk: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    seed: int


PREFILL = PrefillWorkload("chunked prefill", 8, 16384, 512, 32, 8, 128, 20267)


def landscape_workload(batch: int, mean_len: int, seed: int = 20266) -> DecodeWorkload:
    """One cell of the decode-throughput landscape over (B, mean context C):
    lengths uniform in [C/2, 3C/2], 32 query / 8 KV heads, head_dim 128 (the
    head geometry of the paper's Qwen3-8B runs)."""
    lo, hi = mean_len // 2, (3 * mean_len) // 2
    return DecodeWorkload(f"landscape B={batch} C={mean_len}", batch, 32, 8, 128, "uniform",
                          (lo, hi), hi, seed + batch * 1000003 + mean_len)


COMPOSITIONS = ("equal", "uniform", "lognormal", "bimodal", "one_giant")


def composition_lengths(batch: int, mean_len: int, composition: str,
                        seed: int = 20269) -> np.ndarray:
    """Context lengths of one resident batch with B * C tokens in total, spread in
    one of five ways (the within-batch composition of the paper's Fig. 4(b)):

    * ``equal``: every trajectory at C;
    * ``uniform``: U[C/2, 3C/2];
    * ``lognormal``: e^{N(0, 1)} rescaled to mean C (heavy-tailed, like response
      lengths);
    * ``bimodal``: one trajectory in 8 holds 9/16 of the tokens (4.5 C each when
      8 divides B), the rest share the other 7/16 (C/2 each);
    * ``one_giant``: one trajectory holds half of all tokens, the others share
      the rest equally.

    Lengths are at least 16; the total is B * C up to rounding (in expectation for
    ``uniform``).
    """
    if batch < 1 or mean_len < 16:
        raise ValueError("need batch >= 1 and mean length >= 16")
    total = batch * mean_len
    rng = np.random.Generator(np.random.PCG64(seed + batch * 1000003 + mean_len))
    if composition == "equal":
        x = np.full(batch, float(mean_len))
    elif composition == "uniform":
        x = rng.integers(mean_len // 2, (3 * mean_len) // 2, size=batch, endpoint=True).astype(float)
    elif composition == "lognormal":
        x = np.exp(rng.normal(0.0, 1.0, size=batch))
        x *= total / x.sum()
    elif composition == "bimodal":
        k = max(1, batch // 8)  # long trajectories, holding 9/16 of the tokens
        x = np.full(batch, total * 7 / 16 / max(batch - k, 1))
        x[rng.permutation(batch)[:k]] = total * 9 / 16 / k if batch > k else total / batch
    elif composition == "one_giant":
        x = np.full(batch, total / 2 / max(batch - 1, 1))
        x[rng.integers(batch)] = total / 2 if batch > 1 else total
    else:
        raise ValueError(f"unknown composition {composition!r}")
    return np.maximum(np.round(x), 16).astype(np.int32)


def composition_workload(batch: int, mean_len: int, composition: str,
                         seed: int = 20269) -> DecodeWorkload:
    """A decode batch (32 query / 8 KV heads, head_dim 128) with the lengths of
    ``composition_lengths``."""
    lens = composition_lengths(batch, mean_len, composition, seed)
    max_len = -(-int(lens.max()) // PAGE_SIZE) * PAGE_SIZE
    return DecodeWorkload(f"composition {composition} B={batch} C={mean_len}", batch, 32, 8, 128,
                          "fixed", tuple(int(n) for n in lens), max_len, seed + 7 * batch + mean_len)


def draw_lengths(kind: str, args: tuple, batch: int,
                 rng: np.random.Generator) -> np.ndarray:
    """Context lengths n_b (int32)."""
    if kind == "fixed":
        if len(args) != batch:
            raise ValueError("fixed lengths need one value per trajectory")
        return np.asarray(args, dtype=np.int32)
    if kind == "uniform":
        lo, hi = args
        return rng.integers(lo, hi, size=batch, endpoint=True).astype(np.int32)
    if kind == "lognormal":
        median, sigma, lo, hi = args
        x = np.round(median * np.exp(rng.normal(0.0, sigma, size=batch)))
        return np.clip(x, lo, hi).astype(np.int32)
    raise ValueError(f"unknown length distribution {kind!r}")


def scatter_block_table(context_lens: np.ndarray, page_size: int, max_pages: int,
                        pool_pages: int | None, rng: np.random.Generator):
    """Assign each trajectory's logical pages to physical pages of a shuffled pool.

    The logical pages of trajectories 0, 1, ... take consecutive entries of one
    seeded permutation of the pool, so physical pages are fragmented.  Unused
    table entries are -1.  Returns (block_table int32 [B, max_pages], pool_pages).
    """
    pages = -(-context_lens.astype(np.int64) // page_size)
    used = int(pages.sum())
    if pool_pages is None:
        pool_pages = max(used, 1)
    if used > pool_pages:
        raise ValueError(f"batch needs {used} pages, pool has {pool_pages}")
    if pages.max(initial=0) > max_pages:
        raise ValueError("a trajectory is longer than the block table")
    perm = rng.permutation(pool_pages).astype(np.int32)
    table = np.full((len(context_lens), max_pages), -1, dtype=np.int32)
    pos = 0
    for b, p in enumerate(pages):
        table[b, :p] = perm[pos:pos + p]
        pos += p
    return table, pool_pages


def _randn_bf16(shape, gen: torch.Generator, device, scale: float = 1.0):
    x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    if scale != 1.0:
        x.mul_(scale)
    return x.to(torch.bfloat16)


def _randn_bf16_chunked(shape, gen, device, scale=1.0, chunk=1 << 28, out=None):
    """N(0,1)*scale in bf16, drawn in chunks so no full-size fp32 temporary is
    needed; written into ``out`` when given."""
    if out is None:
        out = torch.empty(shape, dtype=torch.bfloat16, device=device)
    flat = out.view(-1)
    for s in range(0, flat.numel(), chunk):
        e = min(s + chunk, flat.numel())
        flat[s:e] = _randn_bf16((e - s,), gen, device, scale)
    return out


@dataclass
class DecodeBatch:
    workload: DecodeWorkload
    context_lens: np.ndarray          # int32 [B]
    block_table: np.ndarray           # int32 [B, max_pages]
    q: torch.Tensor                   # bf16 [B, Hq, D]
    k_pages: torch.Tensor             # bf16 [num_pages, Hkv, P, D]
    v_pages: torch.Tensor             # bf16 [num_pages, Hkv, P, D]
    extra: dict = field(default_factory=dict)

    @property
    def num_pages(self) -> int:
        return self.k_pages.shape[0]


def make_decode_batch(w: DecodeWorkload, device="cpu", seed: int | None = None,
                      batch: int | None = None) -> DecodeBatch:
    """Draw one decode batch for workload ``w`` with values on ``device``.

    ``batch`` overrides the trajectory count (keeping the distribution), which
    the tests use for smaller cases of the same shape.
    """
    seed = w.seed if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    bsz = w.batch if batch is None else batch
    if w.lengths == "fixed" and bsz != w.batch:
        raise ValueError("fixed-length workloads keep their batch size")
    lens = draw_lengths(w.lengths, w.length_args, bsz, rng)
    table, pool_pages = scatter_block_table(lens, w.page_size, w.max_pages,
                                            w.pool_pages, rng)
    gen = torch.Generator(device=device)
    gen.manual_seed(seed)
    q = _randn_bf16((bsz, w.num_q_heads, w.head_dim), gen, device)
    kv_shape = (pool_pages, w.num_kv_heads, w.page_size, w.head_dim)
    k = _randn_bf16_chunked(kv_shape, gen, device, w.k_scale)
    v = _randn_bf16_chunked(kv_shape, gen, device)
    return DecodeBatch(w, lens, table, q, k, v)


def make_prefill_job(w: PrefillWorkload, device="cpu"):
    """The paged pool (fixed lengths, scattered pages), the chunk offsets
    (int64 [batch + 1]) and the queries (bf16 [batch * chunk, Hq, D]) of ``w``."""
    dw = DecodeWorkload(w.name, w.batch, w.num_q_heads, w.num_kv_heads, w.head_dim, "fixed",
                        tuple([w.context] * w.batch), w.context, w.seed)
    b = make_decode_batch(dw, device=device)
    offs = torch.arange(0, (w.batch + 1) * w.chunk, w.chunk, dtype=torch.int64, device=device)
    g = torch.Generator(device=device).manual_seed(w.seed + 1)
    q = torch.randn((w.batch * w.chunk, w.num_q_heads, w.head_dim), generator=g,
                    device=device).to(torch.bfloat16)
    return b, offs, q


@dataclass
class StagingJob:
    workload: StagingWorkload
    context_lens: np.ndarray          # int32 [B]
    block_table: np.ndarray           # int32 [B, max_pages]
    num_pages: int


def make_staging_job(w: StagingWorkload, seed: int | None = None,
                     batch: int | None = None,
                     length_args: tuple | None = None) -> StagingJob:
    """Lengths and block tables of a staging job (values come per layer)."""
    seed = w.seed if seed is None else seed
    rng = np.random.Generator(np.random.PCG64(seed))
    bsz = w.batch if batch is None else batch
    lens = draw_lengths("uniform", length_args or w.length_args, bsz, rng)
    table, pool_pages = scatter_block_table(lens, w.page_size, w.max_pages,
                                            None, rng)
    return StagingJob(w, lens, table, pool_pages)


def fill_layer_pool(out_k: torch.Tensor, out_v: torch.Tensor, seed: int, layer: int):
    """Fill one layer's K and V pages in place with N(0,1) bf16 drawn from
    ``seed * 1000 + layer`` on the tensors' device."""
    gen = torch.Generator(device=out_k.device)
    gen.manual_seed(seed * 1000 + layer)
    _randn_bf16_chunked(out_k.shape, gen, out_k.device, out=out_k)
    _randn_bf16_chunked(out_v.shape, gen, out_v.device, out=out_v)


def bf16_bits(t: torch.Tensor) -> np.ndarray:
    """Raw 16-bit patterns of a bf16 tensor as a numpy uint16 array (host)."""
    if t.dtype != torch.bfloat16:
        raise TypeError("expected a bf16 tensor")
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)
