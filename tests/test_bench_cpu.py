"""Host-side arithmetic of bench.py: the attention time of overlapping launches
(two attention streams) is the length of the union of their event intervals."""
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
