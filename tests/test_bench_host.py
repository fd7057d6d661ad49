"""Host logic of bench.py that needs no GPU: the DRAM-traffic figure is read
from the committed ncu summary only while the decode kernel sources are the
ones that summary names (a stale capture reports null)."""
import bench


def _write(tmp_path, sha, traffic="123456"):
    prof = tmp_path / "profiles"
    prof.mkdir(exist_ok=True)
    (prof / "p.md").write_text(f"# x\n\n- traffic_bytes_per_launch: {traffic}\n- source_sha256: {sha}\n")
    return str(tmp_path)


def test_traffic_is_read_only_for_the_recorded_sources(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _write(tmp_path, "0" * 64))
    monkeypatch.setattr(bench, "decode_source_hash", lambda: "0" * 64)
    assert bench.profiled_traffic("p.md") == 123456
    monkeypatch.setattr(bench, "decode_source_hash", lambda: "1" * 64)
    assert bench.profiled_traffic("p.md") is None
    assert bench.profiled_traffic("missing.md") is None


def test_unparsable_traffic_reads_as_null(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _write(tmp_path, "a" * 64, traffic="n/a"))
    monkeypatch.setattr(bench, "decode_source_hash", lambda: "a" * 64)
    assert bench.profiled_traffic("p.md") is None
