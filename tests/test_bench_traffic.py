"""bench.py's `roofline.traffic` lookup on CPU: a committed ncu record counts
only while the sources of the kernel it captured are unchanged, each record
naming its own source files (the static-chunk and the claimed-group kernels
are built from different files)."""
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture
def bench_in(tmp_path, monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (tmp_path / "profiles").mkdir()
    (tmp_path / "a.cu").write_text("kernel a\n")
    (tmp_path / "b.cuh").write_text("header b\n")
    (tmp_path / "c.cuh").write_text("header c\n")
    return bench, tmp_path


def _write(tmp_path, entries):
    with open(tmp_path / "profiles" / "traffic.json", "w") as f:
        json.dump({"ht_kernel": entries}, f)


def test_record_counts_while_its_own_sources_are_unchanged(bench_in):
    bench, tmp = bench_in
    h_ab = bench.sources_hash(["a.cu", "b.cuh"])
    _write(tmp, {"small": {"dram_bytes_per_launch": 123, "sources": ["a.cu", "b.cuh"],
                           "sources_sha256_16": h_ab}})
    assert bench.profiled_traffic("ht_kernel", "small") == 123
    # a file outside the record's list may change
    (tmp / "c.cuh").write_text("header c, edited\n")
    assert bench.profiled_traffic("ht_kernel", "small") == 123
    # a file of the list may not
    (tmp / "b.cuh").write_text("header b, edited\n")
    assert bench.profiled_traffic("ht_kernel", "small") is None


def test_record_without_a_list_uses_every_kernel_source(bench_in, monkeypatch):
    bench, tmp = bench_in
    monkeypatch.setattr(bench, "HT_KERNEL_SOURCES", ["a.cu", "b.cuh", "c.cuh"])
    _write(tmp, {"big": {"dram_bytes_per_launch": 7,
                         "sources_sha256_16": bench.sources_hash(["a.cu", "b.cuh", "c.cuh"])}})
    assert bench.profiled_traffic("ht_kernel", "big") == 7
    (tmp / "c.cuh").write_text("header c, edited\n")
    assert bench.profiled_traffic("ht_kernel", "big") is None


def test_missing_or_unreadable_records_give_none(bench_in):
    bench, tmp = bench_in
    assert bench.profiled_traffic("ht_kernel", "small") is None  # no file
    _write(tmp, {"small": {"dram_bytes_per_launch": 1, "sources": ["gone.cu"],
                           "sources_sha256_16": "0"}})
    assert bench.profiled_traffic("ht_kernel", "small") is None  # a listed file is missing
    assert bench.profiled_traffic("ht_kernel", "other") is None  # no such workload


def test_committed_records_name_existing_sources():
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        records = json.load(f)["ht_kernel"]
    for name, entry in records.items():
        for p in entry.get("sources", []):
            assert os.path.exists(os.path.join(ROOT, p)), (name, p)
        assert os.path.exists(os.path.join(ROOT, entry["profile"])), name
