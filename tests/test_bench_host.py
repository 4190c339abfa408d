"""Host-side logic of bench.py (no GPU): the kernel-source hash that ties a
committed ncu summary to the code it was taken on, and the lookup of the
summary's DRAM traffic."""
import importlib.util
import os

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _write(path, text):
    with open(path, "w", encoding="utf-8") as f:
        f.write(text)


def test_source_hash_ignores_comments_but_not_code(bench, tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    _write(tmp_path / "k.cu", "// header\nint a = 1;  // trailing\n\nint b = 2;\n")
    h0 = bench.source_hash(["k.cu"])
    _write(tmp_path / "k.cu", "// another header\n// more\nint a = 1;\nint b = 2;   // changed note\n")
    assert bench.source_hash(["k.cu"]) == h0
    _write(tmp_path / "k.cu", "// header\nint a = 1;\nint b = 3;\n")
    assert bench.source_hash(["k.cu"]) != h0
    # file order is part of the hash
    _write(tmp_path / "k.cu", "int a = 1;\nint b = 2;\n")
    _write(tmp_path / "m.cu", "int c = 4;\n")
    assert bench.source_hash(["k.cu", "m.cu"]) != bench.source_hash(["m.cu", "k.cu"])


def test_profiled_traffic_needs_matching_hash(bench, tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    _write(tmp_path / "p.txt", "# comment: ignored\nkernel: k\nsource_hash: abc123\ndram_bytes_per_launch: 1234567\n")
    assert bench.profiled_traffic("p.txt", "abc123") == 1234567.0
    assert bench.profiled_traffic("p.txt", "def456") is None
    assert bench.profiled_traffic("missing.txt", "abc123") is None
    assert bench.profiled_traffic("", "abc123") is None
    _write(tmp_path / "q.txt", "kernel: k\nsource_hash: abc123\n")
    assert bench.profiled_traffic("q.txt", "abc123") is None


def test_committed_summaries_name_their_kernel_sources(bench):
    # every summary the bench can cite exists and carries the fields it reads
    paths = ([bench.SMALL_SUMMARY] + list(bench.READ_SUMMARIES.values()) + list(bench.LM_SUMMARIES.values()) +
             list(bench.TRAIN_SUMMARIES.values()))
    for rel in paths:
        path = os.path.join(ROOT, rel)
        assert os.path.isfile(path), rel
        kv = {}
        for line in open(path, encoding="utf-8"):
            if ":" in line and not line.startswith("#"):
                k, v = line.split(":", 1)
                kv[k.strip()] = v.strip()
        assert len(kv.get("source_hash", "")) == 16, rel
        assert float(kv["dram_bytes_per_launch"]) > 0, rel
