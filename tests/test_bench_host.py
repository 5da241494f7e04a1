"""Host-side pieces of bench.py that need no GPU: the atomic result-file
write (a reader sees the old file or the whole new one)."""
import json
import os

import bench


def test_write_atomic_replaces_whole_file(tmp_path):
    p = tmp_path / "result.json"
    p.write_text("old\n")
    line = json.dumps({"metric": "m", "value": 1.5})
    bench.write_atomic(str(p), line + "\n")
    assert p.read_text() == line + "\n"
    # no temporary file is left beside it
    assert sorted(os.listdir(tmp_path)) == ["result.json"]


def test_write_atomic_failure_leaves_old_file(tmp_path, monkeypatch):
    p = tmp_path / "result.json"
    p.write_text("old\n")

    def boom(src, dst):
        raise OSError("rename failed")

    monkeypatch.setattr(bench.os, "replace", boom)
    try:
        bench.write_atomic(str(p), "new\n")
    except OSError:
        pass
    assert p.read_text() == "old\n"
    assert sorted(os.listdir(tmp_path)) == ["result.json"]
