"""bench.py's host arithmetic, on CPU: the algorithmic bytes of each operation and the traffic record.

The byte counts are the minimum each operation must move (keys 4 B, a row 4 D bytes; B rows per call, U distinct
keys): pull B (4 + row) + U (4 + row); push B (4 + row) + U (4 + 4 row) with replica targets (value and pending
updates read and written), U (4 + 2 row) when every target is main; sync 2 rows per key, 2 per replica and 1 per
refreshed value; create and destroy 3 rows each.
"""
import argparse
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def micro():
    args = argparse.Namespace(batch=1024, zipf=None, span=None, keys=10_000)
    return bench.Micro(args, None)


def counters(**kw):
    base = {k: 0 for k in bench.COUNTERS}
    base.update(kw)
    return base


def test_micro_bytes_per_operation():
    wk = micro()                       # W = 8, D = 64: a row is 256 bytes
    row, W, B = 256, 8, 1024
    d = counters(push_rows=2 * W * B, push_unique=2 * 700, sync_keys=2 * 300, sync_replicas=2 * 500,
                 sync_refreshed=2 * 500, created=2 * 40, destroyed=2 * 30)
    a = bench.alg_bytes_per_step(wk, d, steps=2)
    U = 700
    assert a["push"] == W * B * (4 + row) + U * (4 + 4 * row)
    assert a["push_kernel"] == W * B * (8 + row) + U * (4 + 4 * row)
    assert a["pull"] == W * B * (4 + row) + U * (4 + row)
    assert a["sync"] == 300 * 2 * row + 500 * 3 * row
    assert a["advance"] == (40 + 30) * 3 * row
    assert a["intent"] == W * B * 4 + U * 4


def test_relocation_counts_main_targets_and_versioned_refresh_fewer_writes():
    wk = micro()
    row, W, B = 256, 8, 1024
    d = counters(push_rows=W * B, push_unique=700, sync_keys=300, sync_replicas=500, sync_refreshed=200)
    rep = bench.alg_bytes_per_step(wk, d, steps=1)
    rel = bench.alg_bytes_per_step(wk, d, steps=1, relocate=True)
    assert rep["push"] - rel["push"] == 700 * 2 * row           # 2 rows per distinct key fewer
    assert rep["sync"] == 300 * 2 * row + 500 * 2 * row + 200 * row


def test_traffic_record_only_for_the_captured_source(monkeypatch):
    rec = bench.PUSH_TRAFFIC["mf"]
    rows = 131072
    digest = bench.source_digest([os.path.join(ROOT, p) for p in bench.PUSH_SOURCES])
    got = bench.recorded_traffic("mf", rows)
    if digest == rec["sha256_16"]:
        assert got == pytest.approx(rec["bytes_per_row"] * rows)
    else:
        assert got is None
    monkeypatch.setitem(bench.PUSH_TRAFFIC, "mf", dict(rec, sha256_16="0" * 16))
    assert bench.recorded_traffic("mf", rows) is None
    assert bench.recorded_traffic("micro", rows) is None


def test_source_digest_ignores_comments(tmp_path):
    a = tmp_path / "a.cu"
    b = tmp_path / "b.cu"
    a.write_text("int x = 1;  // one\n\n// a note\nint y = 2;\n")
    b.write_text("int x = 1;\nint y = 2;   // two\n")
    assert bench.source_digest([str(a)]) == bench.source_digest([str(b)])
    b.write_text("int x = 1;\nint y = 3;\n")
    assert bench.source_digest([str(a)]) != bench.source_digest([str(b)])


def test_manager_options_name_every_switch():
    """The `config` of a bench line names the manager's options, the flags turn them off or on, and the
    microbenchmark record keeps them."""
    on = argparse.Namespace(relocate=False, timing="start", delta_refresh=False, no_push_plans=False,
                            pull_staging=False, no_early_events=False)
    off = argparse.Namespace(relocate=True, timing="adaptive", delta_refresh=True, no_push_plans=True,
                             pull_staging=True, no_early_events=True)
    a, b = bench.manager_options(on), bench.manager_options(off)
    assert a["push_plans"] and a["early_events"] and a["placement"] == "replicate" and a["refresh"] == "full"
    assert not b["push_plans"] and not b["early_events"] and b["placement"] == "relocate"
    assert b["action_timing"] == "adaptive" and b["refresh"] == "versioned" and b["pull"] != a["pull"]
    m = bench.micro_args(argparse.Namespace(workload="mf", batch=4, zipf=None, span=2, keys=7, steps=3,
                                            no_early_events=True), 1.4)
    assert m.workload == "micro" and m.zipf == 1.4 and m.batch is None and m.keys is None and m.span is None
    assert m.no_early_events and m.steps == 3
    assert "early_events_per_step" in bench.MICRO_KEYS and "early_advances" in bench.COUNTERS
