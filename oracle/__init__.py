"""fp64 CPU oracle for paged-KV decode attention and prefix staging.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
the CPU-baseline leg of ``bench.py`` may import this package.  It shares no
code with the CUDA path: it never imports ``paper_2609_36899_gb300`` and the
product never imports it.

The arithmetic lives in ``oracle.c`` (plain C, fp64, OpenMP over output rows);
this module only compiles it with gcc and marshals numpy arrays through
ctypes.  bf16 tensors are passed as their raw 16-bit patterns (``uint16``), and
the C code widens each one exactly to double.

Definitions (written out in ``oracle.c``):

* ``decode_attention`` -- one decode step of scaled dot-product attention per
  query head over each trajectory's logical token sequence in a paged KV cache
  (the step the paper identifies as bandwidth-bound, Sec. 2.3 and Sec. 3.1; the
  operator itself comes from the paper's inference backend, Sec. 5).
* ``prefix_stage`` -- the snapshot gather of late-bound KV preparation
  (Sec. 4.4, phase 1).
* ``prefix_load`` -- its inverse, the destination-side materialisation of a
  staged prefix into a paged pool (Sec. 4.4, phase 3).
* ``kv_append`` -- the write of each trajectory's new-token key and value
  into its paged cache that precedes attention in every decode step.
* ``prefill_attention`` -- chunked (re-)prefill attention: each trajectory's
  last C_b tokens attend causally over its paged KV (the fallback of Sec. 4.4
  when prepared KV state cannot be used).

Every function is pinned by the CPU tests in ``tests/test_oracle_*.py``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
SOURCE = _HERE / "oracle.c"
LIBRARY = _HERE / "liboracle.so"

ERRORS = {0: "ok", -1: "invalid argument", -2: "context length out of range",
          -5: "block-table entry out of range"}


class OracleError(RuntimeError):
    pass


def compile_library(source: Path = SOURCE, output: Path = LIBRARY) -> Path:
    """Compile ``source`` with gcc into the shared library ``output``."""
    output = Path(output)
    tmp = output.with_name(output.name + f".tmp{os.getpid()}")
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-std=c11",
           "-o", str(tmp), str(source), "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, output)
    return output


def build() -> Path:
    """Build ``liboracle.so`` next to this file if it is missing or stale."""
    if (not LIBRARY.exists()
            or LIBRARY.stat().st_mtime < SOURCE.stat().st_mtime):
        compile_library()
    return LIBRARY


_P = ctypes.c_void_p
_I64 = ctypes.c_int64


def _ptr(a):
    return None if a is None else ctypes.c_void_p(a.ctypes.data)


def _u16(a) -> np.ndarray:
    a = np.ascontiguousarray(a)
    if a.dtype != np.uint16:
        raise TypeError(f"expected uint16 bf16 bit patterns, got {a.dtype}")
    return a


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


class Oracle:
    """ctypes front end of one compiled copy of ``oracle.c``."""

    def __init__(self, library: str | Path | None = None):
        path = Path(library) if library is not None else build()
        self.lib = ctypes.CDLL(str(path))
        f = self.lib.oracle_decode_attention
        f.restype = ctypes.c_int
        f.argtypes = [_P, _P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64, _I64,
                      _I64, _P, _I64, _P, _P, ctypes.c_int]
        f = self.lib.oracle_prefix_stage
        f.restype = ctypes.c_int
        f.argtypes = [_P, _P, _I64, _I64, _I64, _I64, _I64, _P, _I64, _P, _I64,
                      _I64, _I64, _P, _P, ctypes.c_int]
        f = self.lib.oracle_prefix_load
        f.restype = ctypes.c_int
        f.argtypes = [_P, _P, _I64, _I64, _I64, _I64, _I64, _P, _I64, _P, _I64,
                      _I64, _I64, _P, _P]
        f = self.lib.oracle_prefill_attention
        f.restype = ctypes.c_int
        f.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64, _I64, _I64,
                      _P, _P, ctypes.c_int]
        f = self.lib.oracle_kv_append
        f.restype = ctypes.c_int
        f.argtypes = [_P, _P, _P, _P, _P, _P, _I64, _I64, _I64, _I64, _I64, _I64]
        self.lib.oracle_max_threads.restype = ctypes.c_int

    def max_threads(self) -> int:
        return int(self.lib.oracle_max_threads())

    @staticmethod
    def _check(rc: int):
        if rc != 0:
            raise OracleError(f"oracle returned {rc} ({ERRORS.get(rc, '?')})")

    def decode_attention(self, q, k_pages, v_pages, block_table, context_lens,
                         rows=None, num_threads: int = 0):
        """Attention for one decode token per trajectory.

        q: uint16 [B, Hq, D]; k_pages, v_pages: uint16 [num_pages, Hkv, P, D];
        block_table: int32 [B, max_pages]; context_lens: int32 [B];
        rows: optional int64 array of b * Hq + h to evaluate.
        Returns (out float64 [rows, D] or [B, Hq, D], lse float64).
        """
        q, k_pages, v_pages = _u16(q), _u16(k_pages), _u16(v_pages)
        block_table, context_lens = _i32(block_table), _i32(context_lens)
        batch, hq, d = q.shape
        num_pages, hkv, page, d2 = k_pages.shape
        if d2 != d or v_pages.shape != k_pages.shape:
            raise ValueError("q, k_pages and v_pages disagree on shape")
        if block_table.ndim != 2 or block_table.shape[0] != batch:
            raise ValueError("block_table must be [B, max_pages]")
        max_pages = block_table.shape[1]
        if rows is not None:
            rows = np.ascontiguousarray(rows, dtype=np.int64)
            n_rows = rows.shape[0]
            out = np.empty((n_rows, d), dtype=np.float64)
            lse = np.empty((n_rows,), dtype=np.float64)
        else:
            n_rows = batch * hq
            out = np.empty((batch, hq, d), dtype=np.float64)
            lse = np.empty((batch, hq), dtype=np.float64)
        rc = self.lib.oracle_decode_attention(
            _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
            _ptr(context_lens), batch, hq, hkv, d, page, num_pages, max_pages,
            _ptr(rows), n_rows, _ptr(out), _ptr(lse), int(num_threads))
        self._check(rc)
        return out, lse

    def prefix_stage(self, k_pool, v_pool, block_table, context_lens,
                     layer_begin: int, layer_end: int, dst_offsets=None,
                     dst_size: int | None = None, dst=None, num_threads: int = 0):
        """Gather each trajectory's first n_b tokens of layers
        [layer_begin, layer_end) into contiguous rows.

        k_pool, v_pool: uint16 [L, num_pages, Hkv, P, D].  Returns the uint16
        destination (a new zero-filled array of ``dst_size`` elements, packed
        size by default, unless ``dst`` is given).
        """
        k_pool, v_pool = _u16(k_pool), _u16(v_pool)
        block_table, context_lens = _i32(block_table), _i32(context_lens)
        layers, num_pages, hkv, page, d = k_pool.shape
        if v_pool.shape != k_pool.shape:
            raise ValueError("k_pool and v_pool disagree on shape")
        batch = context_lens.shape[0]
        if dst is None:
            if dst_size is None:
                dst_size = (int(context_lens.astype(np.int64).sum())
                            * (layer_end - layer_begin) * 2 * hkv * d)
            dst = np.zeros(dst_size, dtype=np.uint16)
        if dst_offsets is not None:
            dst_offsets = np.ascontiguousarray(dst_offsets, dtype=np.int64)
        rc = self.lib.oracle_prefix_stage(
            _ptr(k_pool), _ptr(v_pool), layers, num_pages, hkv, page, d,
            _ptr(block_table), block_table.shape[1], _ptr(context_lens), batch,
            layer_begin, layer_end, _ptr(dst), _ptr(dst_offsets), int(num_threads))
        self._check(rc)
        return dst

    def prefix_load(self, k_pool, v_pool, block_table, context_lens,
                    layer_begin: int, layer_end: int, src, src_offsets=None):
        """Write staged rows ``src`` back into ``k_pool`` / ``v_pool`` in place."""
        if k_pool.dtype != np.uint16 or not k_pool.flags.c_contiguous:
            raise TypeError("k_pool must be a C-contiguous uint16 array")
        if v_pool.dtype != np.uint16 or not v_pool.flags.c_contiguous:
            raise TypeError("v_pool must be a C-contiguous uint16 array")
        src = _u16(src)
        block_table, context_lens = _i32(block_table), _i32(context_lens)
        layers, num_pages, hkv, page, d = k_pool.shape
        if src_offsets is not None:
            src_offsets = np.ascontiguousarray(src_offsets, dtype=np.int64)
        rc = self.lib.oracle_prefix_load(
            _ptr(k_pool), _ptr(v_pool), layers, num_pages, hkv, page, d,
            _ptr(block_table), block_table.shape[1], _ptr(context_lens),
            context_lens.shape[0], layer_begin, layer_end, _ptr(src),
            _ptr(src_offsets))
        self._check(rc)
        return k_pool, v_pool

    def kv_append(self, k_pages, v_pages, k_new, v_new, block_table, context_lens):
        """Write the new token's K/V rows (uint16 [B, Hkv, D]) into ``k_pages`` /
        ``v_pages`` (uint16 [num_pages, Hkv, P, D], C-contiguous) in place."""
        for name, a in (("k_pages", k_pages), ("v_pages", v_pages)):
            if a.dtype != np.uint16 or not a.flags.c_contiguous:
                raise TypeError(f"{name} must be a C-contiguous uint16 array")
        k_new, v_new = _u16(k_new), _u16(v_new)
        block_table, context_lens = _i32(block_table), _i32(context_lens)
        num_pages, hkv, page, d = k_pages.shape
        if k_new.shape != (context_lens.shape[0], hkv, d) or v_new.shape != k_new.shape:
            raise ValueError("k_new / v_new must be [B, Hkv, D]")
        rc = self.lib.oracle_kv_append(
            _ptr(k_pages), _ptr(v_pages), _ptr(k_new), _ptr(v_new), _ptr(block_table),
            _ptr(context_lens), context_lens.shape[0], hkv, d, page, num_pages,
            block_table.shape[1])
        self._check(rc)
        return k_pages, v_pages

    def prefill_attention(self, q, q_offsets, k_pages, v_pages, block_table, context_lens,
                          num_threads: int = 0):
        """Causal attention of each trajectory's last C_b tokens.

        q: uint16 [T, Hq, D] (T = q_offsets[-1]); q_offsets: int64 [B + 1].
        Returns (out float64 [T, Hq, D], lse float64 [T, Hq]).
        """
        q, k_pages, v_pages = _u16(q), _u16(k_pages), _u16(v_pages)
        q_offsets = np.ascontiguousarray(q_offsets, dtype=np.int64)
        block_table, context_lens = _i32(block_table), _i32(context_lens)
        total, hq, d = q.shape
        num_pages, hkv, page, d2 = k_pages.shape
        batch = context_lens.shape[0]
        if d2 != d or q_offsets.shape != (batch + 1,) or q_offsets[-1] != total:
            raise ValueError("inconsistent prefill shapes")
        out = np.empty((total, hq, d), dtype=np.float64)
        lse = np.empty((total, hq), dtype=np.float64)
        rc = self.lib.oracle_prefill_attention(
            _ptr(q), _ptr(q_offsets), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
            _ptr(context_lens), batch, hq, hkv, d, page, num_pages, block_table.shape[1],
            _ptr(out), _ptr(lse), int(num_threads))
        self._check(rc)
        return out, lse


_DEFAULT: Oracle | None = None


def default() -> Oracle:
    global _DEFAULT
    if _DEFAULT is None:
        _DEFAULT = Oracle()
    return _DEFAULT


def decode_attention(*args, **kwargs):
    return default().decode_attention(*args, **kwargs)


def prefix_stage(*args, **kwargs):
    return default().prefix_stage(*args, **kwargs)


def prefix_load(*args, **kwargs):
    return default().prefix_load(*args, **kwargs)


def kv_append(*args, **kwargs):
    return default().kv_append(*args, **kwargs)


def prefill_attention(*args, **kwargs):
    return default().prefill_attention(*args, **kwargs)
