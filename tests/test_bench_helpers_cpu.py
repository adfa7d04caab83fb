"""bench.py's host-side helpers on the CPU: the layer chunking of the 48-layer
staging job, the algorithmic byte count of a decode step, and the reading of a
committed ncu summary (a figure is used only while the kernel source it was
taken on is unchanged)."""
import hashlib
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

GB = 1 << 30


def test_staging_chunks_are_the_largest_divisor_that_fits():
    layer = 19 * GB                      # pool + staged rows of one layer
    assert bench.staging_chunk_layers(layer // 2, layer // 2, 280 * GB) == 12
    assert bench.staging_chunk_layers(layer // 2, layer // 2, 200 * GB) == 8
    assert bench.staging_chunk_layers(layer // 2, layer // 2, 30 * GB) == 1
    for free in (25, 60, 90, 150, 230, 300):
        lc = bench.staging_chunk_layers(layer // 2, layer // 2, free * GB)
        assert 48 % lc == 0 and lc * layer <= 0.9 * free * GB


def test_staging_chunks_refuse_when_one_layer_does_not_fit():
    try:
        bench.staging_chunk_layers(10 * GB, 10 * GB, 15 * GB)
    except RuntimeError:
        return
    raise AssertionError("expected a refusal")


def test_decode_bytes_counts_each_token_once_per_kv_head():
    lens = np.array([16, 17, 0], dtype=np.int32)
    hq, hkv, d = 8, 2, 128
    kv = 2 * hkv * d * 2 * int(lens.sum())          # K and V, bf16
    qo = 2 * 3 * hq * d * 2                         # q and out, bf16
    lse = 4 * 3 * hq
    table = 4 * (1 + 2 + 0)                         # entries read: ceil(n / 16)
    assert bench.decode_bytes(lens, hq, hkv, d) == kv + qo + lse + table + 4 * 3


def test_profiled_traffic_follows_the_kernel_source(tmp_path):
    src = tmp_path / "kernel.cu"
    src.write_text("__global__ void k() {}\n")
    digest = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    summary = tmp_path / "profile.md"
    summary.write_text(f"kernel_source_sha256_16: {digest}\n"
                       "dram_bytes_per_launch: 1.5e9\n"
                       "dram_bytes_per_staged_byte: 2.0001\n")
    assert bench.profiled_traffic(str(summary), str(src)) == 1.5e9
    assert bench.profiled_traffic(str(summary), str(src),
                                  key="dram_bytes_per_staged_byte") == 2.0001
    src.write_text("__global__ void k() { /* changed */ }\n")
    assert bench.profiled_traffic(str(summary), str(src)) is None
    assert bench.profiled_traffic(str(tmp_path / "missing.md"), str(src)) is None


def test_reference_arm_prints_the_contract_line():
    """``bench.py --impl reference`` (the fp64 oracle on the host cores) prints one
    JSON line carrying the keys the benchmark contract asks of that arm."""
    import json
    import os
    import subprocess
    import sys
    from pathlib import Path
    root = Path(__file__).resolve().parents[1]
    r = subprocess.run([sys.executable, str(root / "bench.py"), "--impl", "reference",
                        "--workload", "tiny", "--steps", "3", "--warmup", "3",
                        "--reference-seconds", "1"],
                       capture_output=True, text=True, timeout=300, cwd=root,
                       env={**os.environ, "CUDA_VISIBLE_DEVICES": ""})
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["unit"] == "GB/s" and line["value"] > 0
    assert line["higher_is_better"] is True and line["steps"] == 3 and line["warmup"] == 3
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] >= 1
    assert line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    assert line["config"]["workload"] == "tiny decode attention"
