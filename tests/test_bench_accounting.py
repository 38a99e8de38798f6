"""Host-side accounting of bench.py (no GPU): the roofline's algorithmic bytes per frame,
the stored ncu traffic and its staleness rule, and the replicas' disjoint inputs."""
import os
import re
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402
from paper_2609_37007_gb300.synth import MCD  # noqa: E402


def test_algorithmic_bytes_of_one_frame():
    # one frame of 3 calls: the backbone once per call, the heads each call streams, K/V
    # rows attended or written (fp32, 5 layers x 8 KV heads x 128 x K and V), rows fed
    backbone = 5 * (4096 * 1024 + 1024 * 2048 + 6144 * 1024 + 1024 * 3072) * 2
    assert backbone == 157_286_400
    head = 2048 * 1024 * 2
    st = np.zeros(8, dtype=np.int32)
    st[0], st[5], st[6], st[7] = 3, 9, 20, 11            # calls, heads_read, kv_rows, rows_fed
    got = bench.algorithmic_bytes(MCD, st, backbone, head)
    kv_row = 5 * 8 * 128 * 4 * 2
    assert kv_row == 40_960
    assert got == 3 * backbone + 9 * head + 20 * kv_row + 11 * 1024 * 2


def test_algorithmic_bytes_add_over_frames():
    rng = np.random.default_rng(3)
    st = rng.integers(0, 50, size=(7, 8)).astype(np.int32)
    whole = bench.algorithmic_bytes(MCD, st, 1000, 10)
    assert whole == sum(bench.algorithmic_bytes(MCD, st[i], 1000, 10) for i in range(7))


def _profile_fields():
    text = open(bench.PROFILE).read()
    return {k: re.search(k + r"=([0-9a-f]+)", text).group(1)
            for k in ("dram_bytes", "algorithmic_bytes", "source_sha256")}


def test_stored_traffic_scales_the_captured_ratio():
    f = _profile_fields()
    ratio = int(f["dram_bytes"]) / int(f["algorithmic_bytes"])
    assert 0.9 < ratio < 1.5                       # weights read about once per call
    traffic, note = bench.stored_traffic(f["source_sha256"], 2.0e9)
    assert traffic == pytest.approx(ratio * 2.0e9)
    assert "ncu" in note


def test_stored_traffic_is_null_for_other_kernel_sources():
    traffic, note = bench.stored_traffic("0" * 64, 2.0e9)
    assert traffic is None and "changed" in note


def test_replicas_decode_disjoint_frames():
    firsts = [bench.replica_first_frame(r) for r in range(8)]
    assert len(set(firsts)) == 8
    assert all(b - a >= 1_000_000 for a, b in zip(firsts, firsts[1:]))
