"""The algorithmic byte counts behind bench.py's GB/s and roofline figures,
against the counts worked out by hand for the benchmark configurations
(codes + scale/min of every cached token and KV head, bf16 query, fp32
output; a cache write reads bf16 K and V and writes the records)."""
import bench

H_KV, H_Q = 8, 32


def test_record_sizes():
    # 32 + 32 code bytes + 16 + 16 metadata bytes; the compact G = 128 record
    # keeps one (scale, min) pair per token and kind: 4 + 4 bytes
    assert bench.record_bytes(32) == 96
    assert bench.record_bytes(128) == 72
    assert 16 * bench.record_bytes(128) == 1152  # one (page, KV head) record


def test_decode_bytes_of_the_benchmark_shapes():
    # tiny: batch 1 x 1024 tokens
    assert bench.decode_bytes([1024], H_KV, H_Q) == 1024 * 8 * 96 + 8192 + 16384 == 811_008
    # Qwen3-8B-shaped decode: batch 16 x 8192 tokens
    assert bench.decode_bytes([8192] * 16, H_KV, H_Q) == 101_056_512
    # long context: batch 1 x 131072 tokens
    assert bench.decode_bytes([131072], H_KV, H_Q) == 100_687_872
    # the partial kernel's own stream: records only
    assert bench.decode_stream_bytes([8192] * 16, H_KV) == 100_663_296


def test_append_bytes_of_the_prefill():
    # 4 x 32768 tokens x 8 KV heads: 512 B of bf16 K and V read and a
    # 96-byte record written per token and head
    assert bench.append_bytes(4 * 32768, H_KV) == 637_534_208
    assert bench.append_bytes(1, H_KV, 128) == 8 * (512 + 72)


def test_window_split():
    # positions s < sink and s >= n - recent are BF16 window tokens
    assert bench.window_split(1000, 64, 256) == (680, 320)
    assert bench.window_split(320, 64, 256) == (0, 320)
    assert bench.window_split(100, 64, 256) == (0, 100)
    assert bench.window_split(50, 64, 256) == (0, 50)
    assert bench.window_split(1000, 0, 0) == (1000, 0)
    # a windowed decode counts 512 B (bf16 K and V rows) per window token
    got = bench.decode_bytes_win([1000], H_KV, H_Q, 64, 256)
    assert got == 680 * 8 * 96 + 320 * 8 * 512 + 8192 + 16384
    assert bench.decode_bytes_win([1000], H_KV, H_Q, 0, 0) == bench.decode_bytes([1000], H_KV, H_Q)
