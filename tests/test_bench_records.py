"""bench.py reports a kernel's DRAM traffic only from a committed ncu record
taken on the current kernel source, and scales the top-K record per row."""
import importlib.util
import json
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def load_bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_traffic_needs_the_current_source(monkeypatch):
    b = load_bench()
    with open(os.path.join(ROOT, "profiles", "row_kernel_traffic.json")) as fh:
        rec = json.load(fh)
    with open(os.path.join(ROOT, "profiles", "topk_traffic.json")) as fh:
        tk = json.load(fh)
    workload = next(iter(rec["bytes_per_launch"]))
    topk_sources = list(b.TOPK_KERNEL_SOURCES)
    monkeypatch.setattr(b, "source_hash",
                        lambda sources=None: tk["source_hash"] if sources == topk_sources else rec["source_hash"])
    assert b.committed_traffic(workload) == rec["bytes_per_launch"][workload]
    assert b.committed_traffic(workload, 1000, "topk") == tk["bytes_per_row"] * 1000
    monkeypatch.setattr(b, "source_hash", lambda sources=None: "0" * 16)
    assert b.committed_traffic(workload) is None
    assert b.committed_traffic(workload, 1000, "topk") is None


def test_source_hash_covers_the_kernel_sources():
    b = load_bench()
    h = b.source_hash()
    assert len(h) == 16 and h == b.source_hash(b.ROW_KERNEL_SOURCES)
    assert b.source_hash(b.TOPK_KERNEL_SOURCES) != h
    for rel in b.ROW_KERNEL_SOURCES + b.TOPK_KERNEL_SOURCES:
        assert os.path.exists(os.path.join(ROOT, rel)), rel


def test_peak_falls_back_without_the_measured_file(monkeypatch, tmp_path):
    b = load_bench()
    monkeypatch.setattr(b, "ROOT", str(tmp_path))
    assert b.load_peaks() == (6800.0, "fallback")
    (tmp_path / "MEASURED_PEAKS.json").write_text(json.dumps({"hbm_gbs": 6792.1}))
    assert b.load_peaks() == (6792.1, "measured")
