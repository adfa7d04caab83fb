"""ctypes binding of libcadkv.so (argument marshalling only).

Every function here checks tensor dtypes, shapes and devices, allocates
outputs and workspace with torch when the caller gives none, and calls the C
entry point of the same name on the current CUDA stream.  All computation
runs in the library's CUDA kernels; there is no CPU fallback.  If the library
has not been built, the first call raises ``LibraryMissing``.
"""
from __future__ import annotations

import ctypes
import re
from pathlib import Path

import torch

PKG = Path(__file__).resolve().parent
LIBRARY_PATH = PKG / "libcadkv.so"
HEADER_PATH = PKG.parent / "include" / "cadkv.h"

STATUS = {
    "CADKV_OK": 0, "CADKV_ERR_INVALID": -1, "CADKV_ERR_SHAPE": -2, "CADKV_ERR_CUDA": -3,
    "CADKV_ERR_UNSUPPORTED": -4, "CADKV_ERR_OOB": -5, "CADKV_ERR_TIMEOUT": -6,
    "CADKV_ERR_WORKSPACE": -7,
}
PAGE_SIZE = 16


class LibraryMissing(ImportError):
    pass


class CadkvError(RuntimeError):
    def __init__(self, func: str, status: int):
        self.status = status
        super().__init__(f"{func} failed: {status} ({kv_status_string(status)})")


_P = ctypes.c_void_p
_I = ctypes.c_int
_SZ = ctypes.c_size_t

_SIGNATURES = {
    "kv_status_string": (ctypes.c_char_p, [_I]),
    "cadkv_abi_version": (_I, []),
    "cadkv_device_sms": (_I, []),
    "kv_pool_create": (_I, [ctypes.POINTER(_P), _I, _I, _I, _I, _I, _P, _P]),
    "kv_pool_destroy": (_I, [_P]),
    "kv_pool_layer": (_I, [_P, _I, ctypes.POINTER(_P), ctypes.POINTER(_P)]),
    "kv_pool_geometry": (_I, [_P] + [ctypes.POINTER(_I)] * 5),
    "decode_attention_workspace_size": (_SZ, [_I, _I, _I, _I, _I]),
    "decode_attention": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I,
                              _P, _SZ, _P]),
    "decode_attention_split": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I,
                                    _I, _I, _P, _SZ, _P]),
    "decode_attention_plan": (_I, [_P, _P, _P, _I, _I, _I, _I, _I, _I, _P, _SZ, _P]),
    "decode_attention_run": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I,
                                  _P, _SZ, _P]),
    "decode_attention_status": (_I, [_P, _P]),
    "decode_attention_append": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I,
                                     _I, _I, _P, _SZ, _P]),
    "decode_attention_noalloc": (_I, [_P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I,
                                      _P]),
    "decode_attention_noalloc_status": (_I, [_P]),
    "kv_prefix_stage_workspace_size": (_SZ, [_I]),
    "kv_prefix_stage": (_I, [_P, _P, _I, _P, _I, _I, _I, _P, _P, _P, _SZ, _P]),
    "kv_prefix_load": (_I, [_P, _P, _I, _P, _I, _I, _I, _P, _P, _P, _SZ, _P]),
    "kv_prefix_stage_status": (_I, [_P, _P]),
    "cadkv_hbm_read_probe": (_I, [_P, _SZ, _P, _P]),
    "prefill_attention_workspace_size": (_SZ, [_I]),
    "prefill_attention": (_I, [_P, _P, _P, _P, _P, _P, _P, _P, _I, _I, _I, _I, _I, _I, _I, _I,
                               _P, _SZ, _P]),
    "prefill_attention_status": (_I, [_P, _P]),
    "cadkv_wait_selftest": (_I, [ctypes.c_longlong, _P, _SZ, _P]),
}

_lib = None


def library():
    """Load (once) and return the ctypes handle of libcadkv.so."""
    global _lib
    if _lib is None:
        if not LIBRARY_PATH.exists():
            raise LibraryMissing(
                f"{LIBRARY_PATH} is not built; run `python -m paper_2609_36899_gb300.build` "
                "(needs nvcc with sm_103a support)")
        lib = ctypes.CDLL(str(LIBRARY_PATH))
        for name, (res, args) in _SIGNATURES.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
    return _lib


def header_functions() -> list[str]:
    """Names of the functions include/cadkv.h declares."""
    text = HEADER_PATH.read_text()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b([a-z_][a-z0-9_]*)\s*\(", text)) - {"if", "sizeof"})


def kv_status_string(status: int) -> str:
    return library().kv_status_string(int(status)).decode()


def _check(func: str, rc: int):
    if rc != 0:
        raise CadkvError(func, rc)


def _ptr(t):
    # a plain int: the c_void_p argtypes convert it (cheaper than a c_void_p object)
    return None if t is None else t.data_ptr()


def _stream(stream, device):
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def _need(t: torch.Tensor, name: str, dtype, ndim: int | None = None, device=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if ndim is not None and t.dim() != ndim:
        raise ValueError(f"{name} must have {ndim} dims, got {tuple(t.shape)}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


# ------------------------------------------------------------------ decode


def decode_attention_workspace_size(batch: int, num_q_heads: int, num_kv_heads: int,
                                    head_dim: int, max_pages: int) -> int:
    return int(library().decode_attention_workspace_size(batch, num_q_heads, num_kv_heads,
                                                         head_dim, max_pages))


def _decode_args(q, k_pages, v_pages, block_table, context_lens):
    _need(q, "q", torch.bfloat16, 3)
    dev = q.device
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(block_table, "block_table", torch.int32, 2, dev)
    _need(context_lens, "context_lens", torch.int32, 1, dev)
    batch, hq, d = q.shape
    num_pages, hkv, page, d2 = k_pages.shape
    if v_pages.shape != k_pages.shape or d2 != d:
        raise ValueError("k_pages/v_pages must be [num_pages, Hkv, 16, D] matching q")
    if block_table.shape[0] != batch or context_lens.shape[0] != batch:
        raise ValueError("block_table and context_lens must have one row per trajectory")
    return batch, hq, hkv, d, page, num_pages, block_table.shape[1]


def _outputs(q, out, lse, want_lse, workspace, batch, hq, hkv, d, max_pages):
    if out is None:
        out = torch.empty_like(q)
    else:
        _need(out, "out", torch.bfloat16, 3, q.device)
        if out.shape != q.shape:
            raise ValueError("out must have q's shape")
    if lse is None and want_lse:
        lse = torch.empty((batch, hq), dtype=torch.float32, device=q.device)
    elif lse is not None:
        _need(lse, "lse", torch.float32, 2, q.device)
    if workspace is None:
        need = decode_attention_workspace_size(batch, hq, hkv, d, max_pages)
        workspace = torch.empty(max(need, 1), dtype=torch.uint8, device=q.device)
    else:
        _need(workspace, "workspace", torch.uint8, 1, q.device)
    return out, lse, workspace


def decode_attention(q, k_pages, v_pages, block_table, context_lens, out=None, lse=None,
                     workspace=None, slice_pages: int = 0, want_lse: bool = True,
                     stream=None):
    """One decode step of paged-KV attention; returns (out, lse).

    q bf16 [B, Hq, D]; k_pages, v_pages bf16 [num_pages, Hkv, 16, D];
    block_table int32 [B, max_pages]; context_lens int32 [B] (all on one GPU).
    ``slice_pages`` > 0 forces the work-slice length (tests of split invariance).
    """
    batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
        q, k_pages, v_pages, block_table, context_lens)
    out, lse, workspace = _outputs(q, out, lse, want_lse, workspace, batch, hq, hkv, d,
                                   max_pages)
    rc = library().decode_attention_split(
        _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(block_table), _ptr(context_lens),
        _ptr(out), _ptr(lse), batch, hq, hkv, d, page, num_pages, max_pages,
        int(slice_pages), _ptr(workspace), workspace.numel(), _stream(stream, q.device))
    _check("decode_attention", rc)
    return out, lse


class DecodeStep:
    """decode_attention over fixed buffers, validated and marshalled once.

    A serving loop calls decode attention on the same buffers step after step
    (the values change, the tensors do not).  This object checks the tensors
    once, keeps references to them, and each call passes the stored pointers
    straight to the C entry point, so a step costs the host little more than
    the library's own launch work.  Calling it after any of the tensors was
    resized or reallocated is an error the object cannot see: build a new one.
    """

    def __init__(self, q, k_pages, v_pages, block_table, context_lens, out, lse, workspace,
                 slice_pages: int = 0, stream=None, launch: str = "both"):
        """launch: "both" (decode_attention: plan and attention), "plan" or
        "run" (decode_attention_plan / decode_attention_run alone, e.g. one
        plan per decode step and one run per layer)."""
        batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
            q, k_pages, v_pages, block_table, context_lens)
        out, lse, workspace = _outputs(q, out, lse, lse is not None, workspace, batch, hq, hkv,
                                       d, max_pages)
        self.tensors = (q, k_pages, v_pages, block_table, context_lens, out, lse, workspace)
        st = _stream(stream, q.device)
        lib = library()
        if launch == "plan":
            self._name, self._fn = "decode_attention_plan", lib.decode_attention_plan
            self._args = (_ptr(context_lens), _ptr(out), _ptr(lse), batch, hq, hkv, d,
                          max_pages, int(slice_pages), _ptr(workspace), workspace.numel(), st)
            return
        head = (_ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(block_table), _ptr(context_lens),
                _ptr(out), _ptr(lse), batch, hq, hkv, d, page, num_pages, max_pages)
        if launch == "run":
            self._name, self._fn = "decode_attention_run", lib.decode_attention_run
            self._args = head + (_ptr(workspace), workspace.numel(), st)
        elif launch == "both":
            self._name, self._fn = "decode_attention", lib.decode_attention_split
            self._args = head + (int(slice_pages), _ptr(workspace), workspace.numel(), st)
        else:
            raise ValueError("launch must be 'both', 'plan' or 'run'")

    def __call__(self):
        rc = self._fn(*self._args)
        if rc != 0:
            raise CadkvError(self._name, rc)


def decode_attention_append(q, k_new, v_new, k_pages, v_pages, block_table, context_lens,
                            out=None, lse=None, workspace=None, want_lse: bool = True,
                            stream=None):
    """The decode step: write the new token's K/V (bf16 [B, Hkv, D]) at position
    n_b - 1 of each trajectory's pages (in place), then attend; returns (out, lse)."""
    batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
        q, k_pages, v_pages, block_table, context_lens)
    for name, t in (("k_new", k_new), ("v_new", v_new)):
        _need(t, name, torch.bfloat16, 3, q.device)
        if tuple(t.shape) != (batch, hkv, d):
            raise ValueError(f"{name} must be [B, Hkv, D]")
    out, lse, workspace = _outputs(q, out, lse, want_lse, workspace, batch, hq, hkv, d,
                                   max_pages)
    rc = library().decode_attention_append(
        _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
        _ptr(context_lens), _ptr(out), _ptr(lse), batch, hq, hkv, d, page, num_pages,
        max_pages, _ptr(workspace), workspace.numel(), _stream(stream, q.device))
    _check("decode_attention_append", rc)
    return out, lse


def decode_attention_plan(q, k_pages, v_pages, block_table, context_lens, out, lse,
                          workspace, slice_pages: int = 0, stream=None):
    """First launch of decode_attention (the planner) alone."""
    batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
        q, k_pages, v_pages, block_table, context_lens)
    rc = library().decode_attention_plan(
        _ptr(context_lens), _ptr(out), _ptr(lse), batch, hq, hkv, d, max_pages,
        int(slice_pages), _ptr(workspace), workspace.numel(), _stream(stream, q.device))
    _check("decode_attention_plan", rc)


def decode_attention_run(q, k_pages, v_pages, block_table, context_lens, out, lse,
                         workspace, stream=None):
    """Second launch of decode_attention (the attention kernel) alone."""
    batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
        q, k_pages, v_pages, block_table, context_lens)
    rc = library().decode_attention_run(
        _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(block_table), _ptr(context_lens),
        _ptr(out), _ptr(lse), batch, hq, hkv, d, page, num_pages, max_pages,
        _ptr(workspace), workspace.numel(), _stream(stream, q.device))
    _check("decode_attention_run", rc)


def decode_attention_status(workspace, stream=None) -> int:
    """Synchronise the stream and return the device status word (0 = ok)."""
    return int(library().decode_attention_status(_ptr(workspace),
                                                 _stream(stream, workspace.device)))


def decode_attention_noalloc(q, k_pages, v_pages, block_table, context_lens, out=None,
                             lse=None, want_lse: bool = True, stream=None):
    """decode_attention using the library's built-in scratch array instead of
    a workspace, for callers that cannot allocate device memory at call time
    (outputs are still allocated here when not given)."""
    batch, hq, hkv, d, page, num_pages, max_pages = _decode_args(
        q, k_pages, v_pages, block_table, context_lens)
    if out is None:
        out = torch.empty_like(q)
    if lse is None and want_lse:
        lse = torch.empty((batch, hq), dtype=torch.float32, device=q.device)
    rc = library().decode_attention_noalloc(
        _ptr(q), _ptr(k_pages), _ptr(v_pages), _ptr(block_table), _ptr(context_lens),
        _ptr(out), _ptr(lse), batch, hq, hkv, d, page, num_pages, max_pages,
        _stream(stream, q.device))
    _check("decode_attention_noalloc", rc)
    return out, lse


def decode_attention_noalloc_status(stream=None, device=None) -> int:
    """Synchronise the stream and return the status word of the last
    decode_attention_noalloc call on the device (0 = ok)."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else device
    return int(library().decode_attention_noalloc_status(_stream(stream, dev)))


def prefill_attention(q, q_offsets, k_pages, v_pages, block_table, context_lens, out=None,
                      lse=None, workspace=None, want_lse: bool = True, stream=None):
    """Causal attention of each trajectory's last C_b tokens over its paged KV.

    q bf16 [T, Hq, D]; q_offsets int64 [B + 1] (device); the rest as in
    decode_attention.  Returns (out [T, Hq, D], lse [T, Hq]).
    """
    _need(q, "q", torch.bfloat16, 3)
    dev = q.device
    _need(q_offsets, "q_offsets", torch.int64, 1, dev)
    _need(k_pages, "k_pages", torch.bfloat16, 4, dev)
    _need(v_pages, "v_pages", torch.bfloat16, 4, dev)
    _need(block_table, "block_table", torch.int32, 2, dev)
    _need(context_lens, "context_lens", torch.int32, 1, dev)
    total, hq, d = q.shape
    num_pages, hkv, page, d2 = k_pages.shape
    batch = context_lens.shape[0]
    if v_pages.shape != k_pages.shape or d2 != d or q_offsets.shape[0] != batch + 1:
        raise ValueError("inconsistent prefill shapes")
    if out is None:
        out = torch.empty_like(q)
    if lse is None and want_lse:
        lse = torch.empty((total, hq), dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = torch.empty(max(int(library().prefill_attention_workspace_size(batch)), 1),
                                dtype=torch.uint8, device=dev)
    rc = library().prefill_attention(
        _ptr(q), _ptr(q_offsets), _ptr(k_pages), _ptr(v_pages), _ptr(block_table),
        _ptr(context_lens), _ptr(out), _ptr(lse), batch, total, hq, hkv, d, page, num_pages,
        block_table.shape[1], _ptr(workspace), workspace.numel(), _stream(stream, dev))
    _check("prefill_attention", rc)
    return out, lse, workspace


def prefill_attention_status(workspace, stream=None) -> int:
    return int(library().prefill_attention_status(_ptr(workspace),
                                                  _stream(stream, workspace.device)))


# ------------------------------------------------------------------ pool + staging


class KVPool:
    """Handle of a ``cadkv_pool``: per-layer K and V page tensors
    ``[num_pages, Hkv, 16, D]`` bf16.  Keeps the tensors alive."""

    def __init__(self, k_layers, v_layers):
        if len(k_layers) != len(v_layers) or not k_layers:
            raise ValueError("need the same non-zero number of K and V layers")
        shape = tuple(k_layers[0].shape)
        dev = k_layers[0].device
        for name, ts in (("k", k_layers), ("v", v_layers)):
            for i, t in enumerate(ts):
                _need(t, f"{name}_layers[{i}]", torch.bfloat16, 4, dev)
                if tuple(t.shape) != shape:
                    raise ValueError("all layers must share one shape")
        self.k_layers, self.v_layers = list(k_layers), list(v_layers)
        self.num_layers = len(k_layers)
        self.num_pages, self.num_kv_heads, self.page_size, self.head_dim = shape
        self.device = dev
        arr = ctypes.c_void_p * self.num_layers
        kp = arr(*[t.data_ptr() for t in self.k_layers])
        vp = arr(*[t.data_ptr() for t in self.v_layers])
        handle = ctypes.c_void_p()
        with torch.cuda.device(dev):
            rc = library().kv_pool_create(ctypes.byref(handle), self.num_layers,
                                          self.num_pages, self.page_size, self.num_kv_heads,
                                          self.head_dim, ctypes.cast(kp, ctypes.c_void_p),
                                          ctypes.cast(vp, ctypes.c_void_p))
        _check("kv_pool_create", rc)
        self.handle = handle

    def close(self):
        if getattr(self, "handle", None) is not None and self.handle.value:
            library().kv_pool_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def layer_pointers(self, layer: int):
        k, v = ctypes.c_void_p(), ctypes.c_void_p()
        _check("kv_pool_layer", library().kv_pool_layer(self.handle, layer, ctypes.byref(k),
                                                        ctypes.byref(v)))
        return k.value, v.value


def kv_prefix_stage_workspace_size(batch: int) -> int:
    return int(library().kv_prefix_stage_workspace_size(batch))


def staged_size(context_lens_host, layer_begin: int, layer_end: int, num_kv_heads: int,
                head_dim: int) -> int:
    """Elements of a packed staging buffer (no offsets) -- a size, not data."""
    total = int(sum(int(n) for n in context_lens_host))
    return total * (layer_end - layer_begin) * 2 * num_kv_heads * head_dim


def _stage_common(fn, name, pool: KVPool, block_table, context_lens, layer_begin, layer_end,
                  rows, offsets, workspace, stream):
    dev = pool.device
    _need(block_table, "block_table", torch.int32, 2, dev)
    _need(context_lens, "context_lens", torch.int32, 1, dev)
    if rows.is_cuda:
        _need(rows, "rows", torch.bfloat16, None, dev)
    else:  # page-locked host rows: the kernel reads or writes them over the link
        if rows.dtype != torch.bfloat16 or not rows.is_contiguous() or not rows.is_pinned():
            raise ValueError("host rows must be a contiguous, pinned bfloat16 tensor")
    if offsets is not None:
        _need(offsets, "offsets", torch.int64, 1, dev)
    batch = context_lens.shape[0]
    if block_table.shape[0] != batch:
        raise ValueError("block_table must have one row per trajectory")
    if workspace is None:
        workspace = torch.empty(max(kv_prefix_stage_workspace_size(batch), 1),
                                dtype=torch.uint8, device=dev)
    rc = fn(pool.handle, _ptr(block_table), block_table.shape[1], _ptr(context_lens), batch,
            layer_begin, layer_end, _ptr(rows), _ptr(offsets), _ptr(workspace),
            workspace.numel(), _stream(stream, dev))
    _check(name, rc)
    return workspace


def kv_prefix_stage(pool: KVPool, block_table, context_lens, layer_begin: int,
                    layer_end: int, dst, dst_offsets=None, workspace=None, stream=None):
    """Gather each trajectory's prefix of layers [layer_begin, layer_end) into ``dst``
    (a CUDA tensor, or a pinned CPU tensor written directly over the CPU-GPU link)."""
    return _stage_common(library().kv_prefix_stage, "kv_prefix_stage", pool, block_table,
                         context_lens, layer_begin, layer_end, dst, dst_offsets, workspace,
                         stream)


def kv_prefix_load(pool: KVPool, block_table, context_lens, layer_begin: int,
                   layer_end: int, src, src_offsets=None, workspace=None, stream=None):
    """Write staged rows ``src`` (CUDA, or pinned CPU) into the pool pages named by
    ``block_table``."""
    return _stage_common(library().kv_prefix_load, "kv_prefix_load", pool, block_table,
                         context_lens, layer_begin, layer_end, src, src_offsets, workspace,
                         stream)


def cadkv_hbm_read_probe(buf, sink, stream=None):
    """Read all of ``buf`` (a CUDA tensor, size a multiple of 16 bytes) and XOR
    it into ``sink`` (an int64 CUDA tensor of one element, zeroed by the caller)."""
    if not buf.is_cuda or not buf.is_contiguous():
        raise ValueError("buf must be a contiguous CUDA tensor")
    _need(sink, "sink", torch.int64, 1, buf.device)
    rc = library().cadkv_hbm_read_probe(_ptr(buf), buf.numel() * buf.element_size(),
                                        _ptr(sink), _stream(stream, buf.device))
    _check("cadkv_hbm_read_probe", rc)


def cadkv_wait_selftest(limit_ns: int, workspace, stream=None):
    """Run the library's timeout path on purpose (see include/cadkv.h); the status
    word in ``workspace`` then reads CADKV_ERR_TIMEOUT."""
    _need(workspace, "workspace", torch.uint8, 1, None)
    rc = library().cadkv_wait_selftest(int(limit_ns), _ptr(workspace), workspace.numel(),
                                       _stream(stream, workspace.device))
    _check("cadkv_wait_selftest", rc)


def kv_prefix_stage_status(workspace, stream=None) -> int:
    return int(library().kv_prefix_stage_status(_ptr(workspace),
                                                _stream(stream, workspace.device)))
