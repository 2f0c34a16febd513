"""The benchmark's roofline arithmetic against hand-computed values: the
time-weighted tensor peak of a mixed layout, the tensor pipe each group takes
on the staged path (the library's E2M1 gate), padded K per group, and the
algorithmic bytes of an activation quantize."""
import os
import sys

import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402

PK = {"bf16": 1899.8}


def test_mixed_peak_is_the_time_weighted_rate():
    # headline: 3072 channels on E4M3 (2x bf16), 1024 on fp16 (1x): 4 / (3 / 3799.6 + 1 / 1899.8)
    ops = bench.linear_ops(8192, 4096, [3072, 1024])
    assert ops == [2 * 8192 * 4096 * 3072, 2 * 8192 * 4096 * 1024]
    assert bench.mixed_peak(ops, [0, 1], PK) == pytest.approx(4 * 3799.6 / 5, rel=1e-12)
    # the 4/8 conv, 179 channels E4M3 and 77 fp16: 256 * 3799.6 / (179 + 2 * 77)
    assert bench.mixed_peak([179.0, 77.0], [0, 1], PK) == pytest.approx(256 * 3799.6 / 333, rel=1e-12)
    # one pipe alone is its own rate; E2M1 at 6x; an empty group is ignored
    assert bench.mixed_peak([5.0, 0.0], [0, 1], PK) == pytest.approx(3799.6)
    assert bench.mixed_peak([1.0, 1.0], [2, 2], PK) == pytest.approx(6 * 1899.8)
    assert bench.mixed_peak([0.0, 0.0], [0, 1], PK) == 1899.8


def test_group_kinds_follow_the_library_gate():
    # <= 4 bits on both sides: E4M3; wider: fp16
    assert bench.group_kinds([4, 8], [4, 8]) == [0, 1]
    assert bench.group_kinds([3, 5], [4, 4]) == [0, 1]
    # E2M1 needs <= 2 bits on both sides, >= 60 % of the padded codes, rows of >= 2048 codes and
    # 240-column tiles padding N by at most 7 %
    assert bench.group_kinds([2, 8], [2, 8], [3072, 1024], 4096) == [2, 1]        # 75 % of the codes
    assert bench.group_kinds([2, 4], [2, 4], [2048, 2048], 4096) == [0, 0]        # 50 %: stays E4M3
    assert bench.group_kinds([1, 4], [1, 4], [4096, 0], 4096) == [2, 0]           # every code
    assert bench.group_kinds([1, 4], [1, 4], [1792, 896], 256) == [0, 0]          # N = 256: two 240-col tiles
    assert bench.group_kinds([2, 8], [2, 8], [640, 128], 3072) == [0, 1]          # rows of 768 codes


def test_padded_codes_and_quantize_bytes():
    # the conv's weight K per group: 9 taps x roundup(count, 32), rounded up to 128
    assert bench.padded_codes([179, 77], 32, 9) == [1792, 896]
    assert bench.padded_codes([3072, 1024]) == [3072, 1024]
    assert bench.padded_codes([0, 333]) == [0, 384]
    # headline quantize: fp16 read + packed codes (3072 x 4 bits + 1024 x 8 bits per row)
    assert bench.quant_bytes(8192, 4096, [3072, 1024], [4, 8]) == 8192 * 4096 * 2 + 8192 * 2560
    assert bench.quant_bytes(8192, 4096, [3072, 1024], [4, 8]) == 88080384


def test_job_throughput_counts_every_replica():
    assert bench.job_tops(275e9, 0.2, 1) == pytest.approx(275e9 / 0.2e-3 / 1e12)
    assert bench.job_tops(275e9, 0.2, 4) == pytest.approx(4 * 275e9 / 0.2e-3 / 1e12)
    assert bench.max_over_ranks(3.5, 1, "cpu") == 3.5
