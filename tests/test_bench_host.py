"""Host-side helpers of bench.py that need no GPU: how the oracle's bounded
sample is cut into concurrent slices, and which records the bench line
reads."""
import os
import sys

import numpy as np
import pytest

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402
import oracle as O  # noqa: E402


@pytest.mark.parametrize("n,k", [(1, 1), (10, 3), (1000, 16), (7, 16), (4096 * 5 + 3, 4)])
def test_slice_cuts_cover_the_range_in_order(n, k):
    cuts = bench.slice_cuts(n, k)
    assert cuts[0] == 0 and cuts[-1] == n
    assert all(a < b for a, b in zip(cuts, cuts[1:]))
    assert len(cuts) - 1 <= k


def test_slice_cuts_fall_on_block_starts():
    parts = [5000, 3, 9000, 4096]
    starts, off = [], 0
    for p in parts:
        starts.extend(range(off, off + p, 4096))
        off += p
    cuts = bench.slice_cuts(sum(parts), 5, starts)
    assert all(c in starts for c in cuts[:-1]) and cuts[-1] == sum(parts)


def test_parts_between_cuts_tensor_parts():
    assert bench.parts_between([5, 10, 7], 0, 22) == [5, 10, 7]
    assert bench.parts_between([5, 10, 7], 3, 17) == [2, 10, 2]
    assert bench.parts_between([5, 10, 7], 5, 15) == [10]
    assert bench.parts_between([5, 10, 7], 6, 6) == []


def test_sliced_int8_oracle_equals_the_whole_round():
    """Cut at codec block starts, the INT8 oracle on slices gives exactly the
    whole round's outputs, so timing it in slices times the same work."""
    rng = np.random.default_rng(3)
    parts = [4096 * 2 + 100, 777, 4096 + 1]
    n = sum(parts)
    g = rng.normal(0, 0.02, n).astype(np.float32)
    v = rng.normal(0, 1e-3, n).astype(np.float32)
    xs = [(g + rng.normal(0, 1e-3, n)).astype(np.float32) for _ in range(3)]
    whole = O.int8_round(g, v, xs, O.F32, parts, 0.85, 1.5, 1.0)
    starts, off = [], 0
    for p in parts:
        starts.extend(range(off, off + p, 4096))
        off += p
    cuts = bench.slice_cuts(n, 3, starts)
    for a, b in zip(cuts, cuts[1:]):
        part = O.int8_round(g[a:b], v[a:b], [x[a:b] for x in xs], O.F32,
                            bench.parts_between(parts, a, b), 0.85, 1.5, 1.0)
        assert np.array_equal(part["g"], whole["g"][a:b])
        assert np.array_equal(part["v"], whole["v"][a:b])


def test_recorded_entries_follow_the_kernel_source(tmp_path, monkeypatch):
    """A traffic record is used only while its kernel's sources hash to the
    recorded value."""
    import json
    (tmp_path / "profiles").mkdir()
    rec = {"w/k": {"kernel_hash": "abc", "dram_bytes_per_launch": 123,
                   "warps_active_pct": 50.0, "measured_on": "case: ncu ..."}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_source_hash", lambda k: "abc")
    assert bench.recorded_traffic("w", "k") == 123
    assert bench.recorded_occupancy("w", "k") == {"warps_active_pct": 50.0,
                                                  "measured_on": "case"}
    assert bench.recorded_entry("w", "other") is None
    monkeypatch.setattr(bench, "kernel_source_hash", lambda k: "changed")
    assert bench.recorded_traffic("w", "k") is None
    assert bench.recorded_occupancy("w", "k") is None


def test_pinned_budget_is_shared_by_the_ranks_on_a_host():
    import bench
    mem = {"host_ram_bytes": 200e9, "mem_available_bytes": 180e9,
           "cgroup_limit_bytes": None}
    assert bench.pinned_budget(mem) == int(90e9)
    assert bench.pinned_budget(mem, 8) == int(90e9 / 8)
    mem["cgroup_limit_bytes"] = 100e9
    assert bench.pinned_budget(mem, 2) == int(25e9)
    assert bench.pinned_budget({}, 4) == 0
