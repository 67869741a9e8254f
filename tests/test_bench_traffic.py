"""bench.py's DRAM-traffic lookup: one capture block per workload in
profiles/<kernel>_traffic.txt, used only while the kernel source still has the
captured sha256, scaled to a launch by its joined tuples."""
import hashlib
import os
import sys

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
import bench  # noqa: E402


def _tree(tmp_path, src_text, blocks):
    (tmp_path / "profiles").mkdir()
    csrc = tmp_path / "paper_2603_08957_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "k.cu").write_text(src_text)
    lines = ["# header comment: workload: not-a-block"]
    for b in blocks:
        lines += [f"{k}: {v}" for k, v in b.items()] + [""]
    (tmp_path / "profiles" / "k_traffic.txt").write_text("\n".join(lines))


def test_blocks_by_workload_and_source(tmp_path, monkeypatch):
    src = "__global__ void k() {}\n"
    sha = hashlib.sha256(src.encode()).hexdigest()
    _tree(tmp_path, src, [
        {"workload": "gnn", "source_sha256": sha, "pairs": 100, "dram_read_bytes": 1000, "dram_write_bytes": 200},
        {"workload": "gnn2", "source_sha256": sha, "pairs": 10, "dram_read_bytes": 5000, "dram_write_bytes": 0},
        {"workload": "mttkrp", "source_sha256": "0" * 64, "pairs": 1, "dram_read_bytes": 1, "dram_write_bytes": 1},
    ])
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.contract_traffic("k", "gnn", 50) == 600.0           # 12 B per pair
    assert bench.contract_traffic("k", "gnn2", 4) == 2000.0          # 500 B per pair
    assert bench.contract_traffic("k", "mttkrp", 1) is None          # another source
    assert bench.contract_traffic("k", "spgemm", 1) is None          # no capture
    assert bench.contract_traffic("other", "gnn", 1) is None         # no file


def test_changed_source_voids_every_block(tmp_path, monkeypatch):
    src = "__global__ void k() {}\n"
    sha = hashlib.sha256(src.encode()).hexdigest()
    _tree(tmp_path, src, [{"workload": "gnn", "source_sha256": sha, "pairs": 1, "dram_read_bytes": 8,
                           "dram_write_bytes": 0}])
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.contract_traffic("k", "gnn", 1) == 8.0
    (tmp_path / "paper_2603_08957_gb300" / "csrc" / "k.cu").write_text(src + "// edited\n")
    assert bench.contract_traffic("k", "gnn", 1) is None
