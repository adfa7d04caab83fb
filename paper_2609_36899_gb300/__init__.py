"""GB300-native paged-KV decode attention and prefix staging (libcadkv).

The decode step of autoregressive rollout -- attention of one new token per
trajectory over that trajectory's paged KV cache -- is the memory-bound step
that the CadenceRL scheduler reshapes (Sec. 2.3, Sec. 3.1 of the paper).
Late-bound KV preparation (Sec. 4.4) stages a departing trajectory's KV
prefix into contiguous memory and loads it back into a destination pool.

This package is a thin ctypes binding over ``libcadkv.so`` (hand-written CUDA
for sm_103a, C ABI in ``include/cadkv.h``).  Build it with
``python -m paper_2609_36899_gb300.build``.
"""
from ._binding import (  # noqa: F401
    STATUS, CadkvError, DecodeStep, KVPool, LibraryMissing, cadkv_hbm_read_probe, cadkv_wait_selftest,
    decode_attention,
    decode_attention_append, decode_attention_noalloc, decode_attention_noalloc_status, decode_attention_plan, decode_attention_run, decode_attention_status,
    decode_attention_workspace_size, header_functions, kv_prefix_load,
    kv_prefix_stage, kv_prefix_stage_status, kv_prefix_stage_workspace_size,
    kv_status_string, library, prefill_attention, prefill_attention_status, staged_size,
)
