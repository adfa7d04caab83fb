"""Plant plausible mistakes in copies of ``oracle/oracle.c`` and check that the
pins catch every one.

Each mutant is a textual substitution inside one function of the oracle's
source.  The mutated copy is compiled with gcc into a temporary directory and
run through all pins of its kind; at least one pin must fail.  If a
substitution no longer matches the source (the oracle was edited), the test
fails so that the mutant list is kept in step with the code.

Every mutant keeps all memory accesses in bounds, so a broken copy can only
give wrong numbers, never crash the test process.
"""
import re

import pytest

import oracle
from _pins import APPEND_PINS, ATTENTION_PINS, PREFILL_PINS, STAGE_PINS

ATT = "oracle_decode_attention"
STAGE = "oracle_prefix_stage"
LOAD = "oracle_prefix_load"
APPEND = "oracle_kv_append"
PREFILL = "oracle_prefill_attention"

MUTANTS = [
    # (id, function, old, new, count) -- count 0 replaces every occurrence
    ("drop_softmax_scale", ATT,
     "const double scale = 1.0 / sqrt((double)head_dim);", "const double scale = 1.0;", 1),
    ("scale_by_d_not_sqrt_d", ATT,
     "1.0 / sqrt((double)head_dim)", "1.0 / (double)head_dim", 1),
    ("gqa_interleaved_heads", ATT,
     "const int64_t g = h / group;", "const int64_t g = h % num_kv_heads;", 1),
    ("query_indexed_by_kv_head", ATT,
     "q + (b * num_q_heads + h) * head_dim", "q + (b * num_q_heads + g) * head_dim", 1),
    ("slot_reversed_for_keys", ATT,
     "const int64_t slot = t % page_size;",
     "const int64_t slot = (page_size - 1) - t % page_size;", 1),
    ("pages_in_reverse_order", ATT,
     "block_table[b * max_pages + t / page_size]",
     "block_table[b * max_pages + ((n + page_size - 1) / page_size - 1 - t / page_size)]", 0),
    ("last_token_dropped", ATT,
     "for (int64_t t = 0; t < n; ++t) {", "for (int64_t t = 0; t + 1 < n; ++t) {", 0),
    ("exponent_sign_flipped", ATT, "exp(s[t] - m)", "exp(m - s[t])", 1),
    ("values_read_from_keys", ATT, "v_pages + ((phys", "k_pages + ((phys", 1),
    ("normalised_by_length", ATT, "o[d] /= l;", "o[d] /= (double)n;", 1),
    ("lse_without_max", ATT, "lse[i] = m + log(l);", "lse[i] = log(l);", 1),
    ("lse_base_two", ATT, "lse[i] = m + log(l);", "lse[i] = m + log2(l);", 1),
    ("empty_lse_zero", ATT, "lse[i] = -INFINITY;", "lse[i] = 0.0;", 1),
    ("stage_k_v_swapped", STAGE, "(kv == 0 ? k_pool : v_pool)", "(kv == 1 ? k_pool : v_pool)", 1),
    ("stage_rows_head_major", STAGE,
     "(((l - layer_begin) * 2 + kv) * num_kv_heads + h)",
     "((h * (layer_end - layer_begin) + (l - layer_begin)) * 2 + kv)", 1),
    ("stage_slot_reversed", STAGE,
     "const int64_t slot = t % page_size;",
     "const int64_t slot = (page_size - 1) - t % page_size;", 1),
    ("stage_wrong_layer", STAGE, "+ l * layer_stride", "+ (l - layer_begin) * layer_stride", 1),
    ("stage_packed_offset_one_layer", STAGE,
     "layers * 2 * num_kv_heads * head_dim", "2 * num_kv_heads * head_dim", 1),
    ("stage_pool_head_reversed", STAGE,
     "pool + ((phys * num_kv_heads + h) * page_size + slot)",
     "pool + ((phys * num_kv_heads + (num_kv_heads - 1 - h)) * page_size + slot)", 1),
    ("stage_dims_reversed", STAGE, "row[t * head_dim + d] = src[d];",
     "row[t * head_dim + d] = src[head_dim - 1 - d];", 1),
    ("load_tokens_reversed", LOAD,
     "memcpy(d, row + t * head_dim", "memcpy(d, row + (n - 1 - t) * head_dim", 1),
    ("load_k_v_swapped", LOAD, "(kv == 0 ? k_pool : v_pool)", "(kv == 1 ? k_pool : v_pool)", 1),
    ("load_pool_head_reversed", LOAD,
     "pool + ((phys * num_kv_heads + h) * page_size + slot)",
     "pool + ((phys * num_kv_heads + (num_kv_heads - 1 - h)) * page_size + slot)", 1),
    ("append_to_first_token", APPEND, "const int64_t t = n - 1;", "const int64_t t = 0;", 1),
    ("append_head_reversed", APPEND,
     "const int64_t src = (b * num_kv_heads + h) * head_dim;",
     "const int64_t src = (b * num_kv_heads + (num_kv_heads - 1 - h)) * head_dim;", 1),
    ("append_k_only", APPEND, "v_pages[dst + d] = v_new[src + d];", "", 1),
    ("append_next_slot", APPEND, "const int64_t slot = t % page_size;",
     "const int64_t slot = (t + 1) % page_size;", 1),
    ("append_v_from_k", APPEND, "v_pages[dst + d] = v_new[src + d];",
     "v_pages[dst + d] = k_new[src + d];", 1),
    ("prefill_excludes_own_token", PREFILL, "const int64_t n = pos + 1;",
     "const int64_t n = pos > 0 ? pos : 1;", 1),
    ("prefill_attends_whole_context", PREFILL, "const int64_t n = pos + 1;",
     "const int64_t n = context_lens[b];", 1),
    ("prefill_chunk_at_start", PREFILL,
     "const int64_t pos = context_lens[b] - chunk + (row - q_offsets[b]);",
     "const int64_t pos = row - q_offsets[b];", 1),
    ("prefill_gqa_interleaved", PREFILL, "const int64_t g = h / group;",
     "const int64_t g = h % num_kv_heads;", 1),
    ("prefill_drop_softmax_scale", PREFILL,
     "const double scale = 1.0 / sqrt((double)head_dim);", "const double scale = 1.0;", 1),
    ("prefill_exponent_sign_flipped", PREFILL, "exp(s[t] - m)", "exp(m - s[t])", 1),
    ("prefill_values_read_from_keys", PREFILL, "v_pages + ((phys", "k_pages + ((phys", 1),
    ("prefill_normalised_by_length", PREFILL, "o[d] /= l;", "o[d] /= (double)n;", 1),
    ("prefill_lse_without_max", PREFILL, "lse[i] = m + log(l);", "lse[i] = log(l);", 1),
    ("prefill_key_slot_reversed", PREFILL,
     "k_pages + ((phys * num_kv_heads + g) * page_size + t % page_size)",
     "k_pages + ((phys * num_kv_heads + g) * page_size + (page_size - 1 - t % page_size))", 1),
    ("prefill_query_of_next_head", PREFILL,
     "q + (row * num_q_heads + h) * head_dim",
     "q + (row * num_q_heads + (h + 1) % num_q_heads) * head_dim", 1),
]


def _function_span(src: str, name: str):
    m = re.search(r"^int " + name + r"\(", src, flags=re.M)
    assert m, f"function {name} not found in oracle.c"
    end = src.index("\n}\n", m.start())
    return m.start(), end


def mutate(src: str, func: str, old: str, new: str, count: int) -> str:
    a, b = _function_span(src, func)
    body = src[a:b]
    assert old in body, f"mutation anchor {old!r} not found in {func}"
    body = body.replace(old, new) if count == 0 else body.replace(old, new, count)
    return src[:a] + body + src[b:]


@pytest.mark.parametrize("mid,func,old,new,count", MUTANTS, ids=[m[0] for m in MUTANTS])
def test_pins_catch_mutant(tmp_path, mid, func, old, new, count):
    src = oracle.SOURCE.read_text()
    path = tmp_path / f"{mid}.c"
    path.write_text(mutate(src, func, old, new, count))
    lib = oracle.compile_library(path, tmp_path / f"lib{mid}.so")
    orc = oracle.Oracle(lib)
    pins = {ATT: ATTENTION_PINS, APPEND: APPEND_PINS, PREFILL: PREFILL_PINS}.get(
        func, STAGE_PINS)
    caught = []
    for pin in pins:
        try:
            pin(orc)
        except (AssertionError, oracle.OracleError, ValueError, FloatingPointError):
            caught.append(pin.__name__)
    assert caught, f"mutant {mid} survived every pin"
