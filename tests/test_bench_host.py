"""Host logic of bench.py that needs no GPU: the source hash that gates each
committed ncu traffic figure follows the code, not its comments, and the
traffic figure is read only while that hash matches."""
import os

import bench


def _tree(tmp_path, text):
    d = tmp_path / "paper_2608_28726_gb300" / "csrc"
    d.mkdir(parents=True, exist_ok=True)
    (d / "k.cu").write_text(text)
    return str(tmp_path)


def test_source_sha_ignores_comments_and_white_space(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _tree(tmp_path, "int f(int x) {\n  return x + 1;\n}\n"))
    a = bench.source_sha(["k.cu"])
    _tree(tmp_path, "// f adds one\nint f(int x) { /* the\n step */ return x + 1;   }\n")
    assert bench.source_sha(["k.cu"]) == a
    _tree(tmp_path, "int f(int x) {\n  return x + 2;\n}\n")
    assert bench.source_sha(["k.cu"]) != a


def test_profiled_traffic_follows_the_source(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "ROOT", _tree(tmp_path, "int g() { return 3; }\n"))
    prof = tmp_path / "p.md"
    prof.write_text("# k\n\n- kernel_source_sha: `%s`\n- dram_bytes_per_launch: `12345`\n"
                    % bench.source_sha(["k.cu"]))
    assert bench.profiled_file_traffic(str(prof), ["k.cu"]) == 12345
    _tree(tmp_path, "int g() { return 4; }\n")
    assert bench.profiled_file_traffic(str(prof), ["k.cu"]) is None
    assert bench.profiled_file_traffic(os.path.join(str(tmp_path), "missing.md"), ["k.cu"]) is None
