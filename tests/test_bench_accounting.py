"""The benchmark's roofline accounting (host arithmetic only, no GPU): algorithmic bytes and
flops of a layer forward at the benchmark shape, and the rule that the ncu traffic figure is
used only while the profiled kernel's source is unchanged."""
import hashlib
import os

import pytest

import bench
from dmoe_synth import LAYER


def test_layer_bytes_at_the_benchmark_shape():
    # one expert = gate + up + down, 3 * 2048 * 512 bf16 values = 6,291,456 B
    expert = 3 * 2048 * 512 * 2
    assert expert == 6_291_456
    # 8 unique experts + the shared one, W_r fp32 [2048, 256], bias, x in and y out
    want = 9 * expert + 2048 * 256 * 4 + 256 * 4 + 2 * 32 * 2048 * 2
    assert bench.layer_bytes(LAYER, 8) == want == 58_983_424
    # the expert launch: weights + x + y, no router
    assert bench.experts_bytes(LAYER, 8) == 9 * expert + 2 * 32 * 2048 * 2 == 56_885_248


def test_layer_flops_at_the_benchmark_shape():
    # 2 flops per multiply-add: 32 tokens x (8 routed + 1 shared) SwiGLU experts, + router
    want = 2 * 32 * 9 * 3 * 2048 * 512 + 2 * 32 * 2048 * 256
    assert bench.layer_flops(LAYER) == want == 1_845_493_760


def test_token_routing_bytes_grow_by_one_expert_per_unique_expert():
    d = bench.layer_bytes(LAYER, 105) - bench.layer_bytes(LAYER, 104)
    assert d == 3 * 2048 * 512 * 2


def test_profile_traffic_needs_the_profiled_source(tmp_path, monkeypatch):
    src_dir = tmp_path / "paper_2605_30876_gb300" / "csrc"
    src_dir.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    src = src_dir / "k.cu"
    src.write_bytes(b"__global__ void k() {}\n")
    h = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (tmp_path / "profiles" / "k_layer_block.txt").write_text(
        f"summary\nsource_sha256_16: {h}   (the kernel's source)\n"
        "dram_bytes_per_launch: 1234567\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_from_profile("k", "k.cu") == pytest.approx(1234567.0)
    # any change to the source voids the figure
    src.write_bytes(b"__global__ void k() { }\n")
    assert bench.traffic_from_profile("k", "k.cu") is None
    # and so does a missing profile
    assert bench.traffic_from_profile("other", "k.cu") is None


def test_committed_expert_profile_names_a_source_hash():
    path = os.path.join(bench.ROOT, "profiles", "moe_decode_layer_block.txt")
    text = open(path).read()
    assert "source_sha256_16:" in text and "dram_bytes_per_launch:" in text
