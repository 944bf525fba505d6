"""Host-side parts of bench.py: the roofline numerator (algorithmic bytes per
stage), the whole-job aggregation and the lookup of committed ncu traffic.
No GPU is used."""
import json
import os

import pytest

import bench
from paper_2411_12364_gb300 import workloads


def test_algorithmic_bytes_of_decode_1m():
    """decode_1m at 64 tokens, worked by hand (bf16, es = 2; H = 2, D_k = 128,
    D_i = 1024, K = 2 * 1024, k = m = 32, D_v = 256, E = 4, D'_v = 1024):
      query   W_q 2*128*1024*2 + x 64*1024*2             = 655,360
      score   keys 2*2*2048*128*2                         = 2,097,152
      select  64*2 * (2*2048*4 + 128*4 + 2*32*128*2 + 32*12) = 4,308,992
      gather  min(64*2*32, 1024^2) rows * 256 * 2         = 2,097,152
      project W_p 4*256*1024*2 + out 64*1024*2            = 2,228,224"""
    b = bench.algorithmic_bytes(workloads.layer_config("decode_1m"), 64)
    assert b == {"query": 655_360, "score": 2_097_152, "select": 4_308_992,
                 "gather": 2_097_152, "project": 2_228_224}


def test_algorithmic_bytes_gather_is_capped_by_the_table():
    """min(B*H*m, N) rows: a batch that would read more rows than the table
    holds reads each row at most once (tiny_fp32: N = 65,536 rows of 1 KB)."""
    cfg = workloads.layer_config("tiny_fp32")
    H, m, N = cfg["heads"], cfg["topm"], cfg["n"] ** 2
    big = N // (H * m) * 4
    assert bench.algorithmic_bytes(cfg, big)["gather"] == N * cfg["d_v"] * 4
    assert bench.algorithmic_bytes(cfg, 16)["gather"] == 16 * H * m * cfg["d_v"] * 4


def test_algorithmic_bytes_with_cores_and_column_query():
    """h = 2 component cores add one fp32 weight per slot; a separate column
    query doubles the query projection's weight and the query read."""
    base = workloads.layer_config("decode_1m")
    b1 = bench.algorithmic_bytes(base, 64)
    b2 = bench.algorithmic_bytes(dict(base, cores=2), 64)
    assert b2["select"] - b1["select"] == 64 * 2 * 32 * 4
    b3 = bench.algorithmic_bytes(dict(base, share_query=0), 64)
    assert b3["query"] - b1["query"] == 2 * 128 * 1024 * 2
    assert b3["select"] - b1["select"] == 64 * 2 * 128 * 4


def test_algorithmic_bytes_with_candidate_lists():
    """With the candidate lists the selection reads each axis' group counts
    (ceil(K/16) x 4 B) and at least k list entries (8 B) instead of the
    axis' K rank-1 keys (4 B each); the other stages are the same."""
    cfg = workloads.layer_config("prefill_16k")
    B, H, k = 16384, cfg["heads"], cfg["topk"]
    K = 2 * cfg["n"]   # E = 4
    b0 = bench.algorithmic_bytes(cfg, B)
    b1 = bench.algorithmic_bytes(cfg, B, lists=True)
    assert b0["select"] - b1["select"] == B * H * 2 * (K * 4 - (K // 16 * 4 + k * 8))
    assert {s: b0[s] for s in b0 if s != "select"} == {s: b1[s] for s in b1 if s != "select"}


def test_aggregate_step_without_ranks():
    ms, value = bench.aggregate_step(0.035, 64)
    assert ms == 0.035
    assert value == pytest.approx(64 / 35e-6)


def test_ncu_traffic_only_for_the_measured_source():
    """The committed DRAM bytes of a stage are reported only for the workload
    and batch they were taken on, and only while the kernel source still has
    the hash they were taken on."""
    path = os.path.join(bench.ROOT, "profiles", "ncu_traffic.json")
    entries = json.load(open(path))
    for stage, e in entries.items():
        src = os.path.join(bench.ROOT, "paper_2411_12364_gb300", "csrc", e["source"])
        same = bench.source_sha(src) == e["source_sha"]
        got = bench.ncu_traffic(stage, e["workload"], int(e["batch"]))
        assert got == (float(e["dram_bytes_per_launch"]) if same else None)
        assert bench.ncu_traffic(stage, e["workload"], int(e["batch"]) + 1) is None
        assert bench.ncu_traffic(stage, "another_workload", int(e["batch"])) is None
    assert bench.ncu_traffic("no_such_stage", "decode_1m", 64) is None
