"""bench.py's ncu traffic records: a record's bytes reach the bench line only while the
sources it lists hash to the value stored beside them, so a kernel edited after its capture
reports no traffic instead of a stale one.  Runs on temporary files, not on the live records."""
import hashlib
import json
import os

import pytest


def _write_record(root, kernel, workload, sources, nbytes, digest=None):
    h = hashlib.sha256()
    for src in sources:
        with open(os.path.join(root, src), "rb") as f:
            h.update(f.read())
    os.makedirs(os.path.join(root, "profiles"), exist_ok=True)
    rec = {kernel: {workload: {"bytes": nbytes, "sources": sources,
                               "sha256_16": digest or h.hexdigest()[:16]}}}
    with open(os.path.join(root, "profiles", "traffic.json"), "w") as f:
        json.dump(rec, f)


@pytest.fixture
def bench_at(tmp_path, monkeypatch):
    import bench
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    for name, text in (("a.cu", "// kernel\n"), ("b.h", "// header\n")):
        (tmp_path / name).write_text(text)
    return bench, tmp_path


def test_record_used_while_sources_match(bench_at):
    bench, root = bench_at
    _write_record(str(root), "k", "w", ["a.cu", "b.h"], 12345)
    assert bench._traffic("k", "w") == 12345


def test_record_dropped_when_a_source_changes(bench_at):
    bench, root = bench_at
    _write_record(str(root), "k", "w", ["a.cu", "b.h"], 12345)
    (root / "b.h").write_text("// header, edited after the capture\n")
    assert bench._traffic("k", "w") is None


def test_record_dropped_when_sources_are_reordered_or_missing(bench_at):
    bench, root = bench_at
    _write_record(str(root), "k", "w", ["a.cu", "b.h"], 12345)
    with open(root / "profiles" / "traffic.json") as f:
        rec = json.load(f)
    rec["k"]["w"]["sources"] = ["b.h", "a.cu"]  # same files, other order: another digest
    with open(root / "profiles" / "traffic.json", "w") as f:
        json.dump(rec, f)
    assert bench._traffic("k", "w") is None
    rec["k"]["w"]["sources"] = ["a.cu", "gone.h"]
    with open(root / "profiles" / "traffic.json", "w") as f:
        json.dump(rec, f)
    assert bench._traffic("k", "w") is None


def test_unknown_kernel_or_workload_has_no_record(bench_at):
    bench, root = bench_at
    _write_record(str(root), "k", "w", ["a.cu"], 7)
    assert bench._traffic("k", "other") is None
    assert bench._traffic("other", "w") is None


def test_live_records_name_existing_sources():
    """Every committed record lists files that exist and a 16-hex-digit digest (whether the
    digest still matches is bench.py's business at run time, not this test's)."""
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    with open(os.path.join(root, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    for kernel, per in rec.items():
        if kernel.startswith("_"):
            continue
        for workload, r in per.items():
            assert r["bytes"] > 0, (kernel, workload)
            assert len(r["sha256_16"]) == 16 and int(r["sha256_16"], 16) >= 0
            for src in r["sources"]:
                assert os.path.exists(os.path.join(root, src)), src
