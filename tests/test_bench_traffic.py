"""The benchmark reports the GEMM class's DRAM traffic from the committed ncu summary only while the
GEMM source it was captured on is unchanged (its sha256 is recorded beside the figure). No GPU."""
import hashlib
import os
import shutil

import bench


def _fake_root(tmp_path, gemm_src: bytes, summary: str):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "gemm_llava15_layer.md").write_text(summary)
    csrc = tmp_path / "paper_2609_34977_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "gemm.cu").write_bytes(gemm_src)
    return str(tmp_path)


def test_committed_summary_matches_the_committed_source():
    # the committed capture is of the committed kernel source: the figure is reported
    t = bench.gemm_traffic()
    assert t is not None and t > 1e8


def test_traffic_is_dropped_once_the_source_changes(tmp_path, monkeypatch):
    src = b"// a kernel\n"
    digest = hashlib.sha256(src).hexdigest()
    summary = f"# capture\n\ntraffic_bytes_per_launch: 123456789\nsource_sha256: {digest}\n"
    monkeypatch.setattr(bench, "ROOT", _fake_root(tmp_path, src, summary))
    assert bench.gemm_traffic() == 123456789.0
    # one byte more in the source: the counters no longer describe it
    with open(os.path.join(bench.ROOT, "paper_2609_34977_gb300", "csrc", "gemm.cu"), "ab") as f:
        f.write(b" ")
    assert bench.gemm_traffic() is None


def test_missing_summary_gives_no_traffic(tmp_path, monkeypatch):
    root = _fake_root(tmp_path, b"x", "no figures here\n")
    monkeypatch.setattr(bench, "ROOT", root)
    assert bench.gemm_traffic() is None
    shutil.rmtree(os.path.join(root, "profiles"))
    assert bench.gemm_traffic() is None
