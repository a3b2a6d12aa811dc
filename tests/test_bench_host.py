"""bench.py on the host: the recorded DRAM traffic is used only while the
sources of the kernel it was captured on are unchanged, kernel by kernel."""
import json
import os
import shutil

import pytest

import bench


@pytest.fixture()
def tree(tmp_path, monkeypatch):
    # a copy of the kernel sources and a traffic record hashed on them
    for rel in {r for srcs in bench.KERNEL_SOURCES.values() for r in srcs}:
        dst = tmp_path / rel
        dst.parent.mkdir(parents=True, exist_ok=True)
        shutil.copy(os.path.join(bench.ROOT, rel), dst)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (tmp_path / "profiles").mkdir()
    rec = {k: {"w": {"dram_bytes_per_launch": 1000 + i, "source_hash": bench.kernel_source_hash(k)}}
           for i, k in enumerate(sorted(bench.KERNEL_SOURCES))}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    return tmp_path


def test_traffic_used_while_sources_match(tree):
    assert bench.recorded_traffic("spec_accept", "w") == 1000
    assert bench.recorded_traffic("verify_attention", "w") == 1001
    assert bench.recorded_traffic("verify_attention", "other-workload") is None


def test_a_change_voids_only_that_kernels_traffic(tree):
    with open(tree / "paper_2607_20507_gb300/csrc/spec_accept.cu", "a") as f:
        f.write("\n// changed\n")
    assert bench.recorded_traffic("spec_accept", "w") is None
    assert bench.recorded_traffic("verify_attention", "w") == 1001
    with open(tree / "paper_2607_20507_gb300/csrc/cs_device.cuh", "a") as f:
        f.write("\n// changed\n")
    assert bench.recorded_traffic("verify_attention", "w") is None


def test_missing_record_reads_as_none(tree):
    os.remove(tree / "profiles" / "traffic.json")
    assert bench.recorded_traffic("verify_attention", "w") is None
