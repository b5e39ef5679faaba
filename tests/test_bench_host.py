"""Host-side arithmetic of bench.py that needs no GPU: the source hash that
keys the stored DRAM traffic to a kernel's code, and the byte counts the
roofline divides by."""
from __future__ import annotations

import pytest

import bench


def _tree(tmp_path, text):
    d = tmp_path / "paper_2606_28560_gb300" / "csrc"
    d.mkdir(parents=True, exist_ok=True)
    (d / "k.cu").write_text(text)


def _sha(tmp_path, monkeypatch, text):
    _tree(tmp_path, text)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    return bench.sources_sha256(("k.cu",))


CODE = "int f(int x) {\n    return x + 1;\n}\n"


def test_source_hash_ignores_comments_and_blank_lines(tmp_path, monkeypatch):
    base = _sha(tmp_path, monkeypatch, CODE)
    commented = ("// header comment\n/* block\n   comment */\nint f(int x) {   // trailing\n\n"
                 "    return x + 1;  \n}\n\n")
    assert _sha(tmp_path, monkeypatch, commented) == base


@pytest.mark.parametrize("changed", ["int f(int x) {\n    return x + 2;\n}\n",
                                     "int f(int x) {\n    return x+1;\n}\n",
                                     "int f(int y) {\n    return y + 1;\n}\n"])
def test_source_hash_follows_code(tmp_path, monkeypatch, changed):
    assert _sha(tmp_path, monkeypatch, changed) != _sha(tmp_path, monkeypatch, CODE)


def test_stored_traffic_is_null_once_code_changes(tmp_path, monkeypatch):
    # a kernel whose hashed sources differ from the capture reports no traffic
    _tree(tmp_path, CODE)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setitem(bench.NCU_TRAFFIC, "probe", {"bytes_at_b32": 3200, "sources": ("k.cu",),
                                                     "sha256": bench.sources_sha256(("k.cu",))})
    assert bench.ncu_traffic("probe") == round(3200 * bench.B / 32)
    _tree(tmp_path, CODE.replace("+ 1", "+ 3"))
    assert bench.ncu_traffic("probe") is None
    assert bench.ncu_traffic("no such kernel") is None


def test_method_bytes_per_query_head():
    # forward Q, K, V, O rows once (512 B per query-head at D = 64, bf16) plus
    # the fp32 lse; the step counts 512 + 1024 B per query-head
    n = bench.B * bench.H * bench.T
    mb = bench.method_bytes()
    assert mb["fwd"] == n * (4 * 128 + 4)
    assert mb["bwd_query_mma"] == n * (6 * 128 + 4)
    assert mb["bwd_key_mma"] == n * 4 * 128
    assert mb["rope_k"] == 0
    assert bench.step_method_bytes() == bench.L * n * (512 + 1024)
