"""Host logic of bench.py that needs no GPU: the DRAM-traffic figure of the
roofline comes from a committed ncu launch list only while the GEMM sources
are the ones that launch list measured."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _profile(tmp_path, sha, nbytes):
    p = tmp_path / "traffic.md"
    p.write_text("# capture\n\n    ncu --metrics ... (command lines are indented and ignored)\n\n"
                 f"- gemm_source_sha16: `{sha}`\n- dram_bytes_per_gemm_launch: `{nbytes}`\n")
    return str(p)


def test_traffic_is_read_while_the_gemm_sources_match(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_PROFILE", _profile(tmp_path, bench.gemm_source_hash(), 123456789))
    value, source = bench.gemm_traffic()
    assert value == 123456789.0 and source.endswith("traffic.md")


def test_traffic_is_null_once_the_gemm_sources_change(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_PROFILE", _profile(tmp_path, "0123456789abcdef", 123456789))
    value, why = bench.gemm_traffic()
    assert value is None and "changed" in why


def test_traffic_without_a_capture_is_null(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_PROFILE", str(tmp_path / "missing.md"))
    value, why = bench.gemm_traffic()
    assert value is None and why == "no capture"


def test_source_hash_covers_every_gemm_source(tmp_path, monkeypatch):
    """Changing any one of the GEMM sources changes the hash (each file is read)."""
    base = bench.gemm_source_hash()
    csrc = tmp_path / "paper_2609_37924_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for f in bench.GEMM_SOURCES:
        (csrc / f).write_bytes(open(os.path.join(ROOT, "paper_2609_37924_gb300", "csrc", f), "rb").read())
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.gemm_source_hash() == base
    seen = {base}
    for f in bench.GEMM_SOURCES:
        orig = (csrc / f).read_bytes()
        (csrc / f).write_bytes(orig + b"\n")
        h = bench.gemm_source_hash()
        assert h not in seen, f
        seen.add(h)
        (csrc / f).write_bytes(orig)
