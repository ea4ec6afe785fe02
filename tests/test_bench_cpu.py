"""Host-side arithmetic of bench.py: the attention time of overlapping launches
(two attention streams) is the length of the union of their event intervals;
the recorded DRAM traffic is weighted by the timed launches' kinds."""
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))

import bench  # noqa: E402


def test_union_of_disjoint_intervals_is_their_sum():
    assert bench.union_length([(0.0, 1.0), (2.0, 3.5)]) == 2.5


def test_overlaps_count_once():
    # block b + 1 starts in block b's tail: [0, 10] and [8, 18] cover 18
    assert bench.union_length([(8.0, 18.0), (0.0, 10.0)]) == 18.0
    # nested and touching intervals
    assert bench.union_length([(0.0, 10.0), (2.0, 3.0), (10.0, 12.0)]) == 12.0


def test_empty_and_single():
    assert bench.union_length([]) == 0.0
    assert bench.union_length([(5.0, 7.0)]) == 2.0


def test_many_overlapping_launches_never_exceed_the_span():
    iv = [(i * 1.0, i * 1.0 + 1.5) for i in range(100)]
    u = bench.union_length(iv)
    assert u == 100.5
    assert u <= sum(b - a for a, b in iv)


def test_recorded_traffic_weights_launch_kinds(tmp_path, monkeypatch):
    """roofline.traffic: the mean of the per-kind DRAM bytes over the timed
    launches' kinds (materialise: a COMPUTE or FULL sample; refresh: a
    BOUNDARY sample; reuse), null once the kernel source no longer matches."""
    import json
    os.makedirs(tmp_path / "profiles")
    for rel in bench.ATTN_SOURCES:
        os.makedirs(os.path.dirname(tmp_path / rel), exist_ok=True)
        (tmp_path / rel).write_text("kernel source " + rel)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    rec = {"source_hash": bench.source_hash(*bench.ATTN_SOURCES),
           "per_launch": {"w": {"materialise": {"bytes": 1000}, "refresh": {"bytes": 700},
                                "reuse": {"bytes": 400}},
                          "old": {"refresh": {"bytes": 700}, "reuse": {"bytes": 400}}}}
    (tmp_path / "profiles" / "attn_traffic.json").write_text(json.dumps(rec))
    modes = [[3], [1], [2, 0], [0], [0, 1]]  # materialise, refresh, materialise, reuse, refresh
    r = bench.recorded_traffic("w", modes)
    assert r["bytes"] == round((2 * 1000 + 2 * 700 + 400) / 5)
    assert r["mix"] == {"materialise_launches": 2, "refresh_launches": 2, "reuse_launches": 1}
    r = bench.recorded_traffic("old", modes)  # a record without the materialise kind
    assert r["bytes"] == round((4 * 700 + 400) / 5)
    assert bench.recorded_traffic("w") is None
    (tmp_path / bench.ATTN_SOURCES[0]).write_text("changed")
    assert bench.recorded_traffic("w", modes) is None
