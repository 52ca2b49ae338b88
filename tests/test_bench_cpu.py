"""Host-side rules of bench.py that decide what its JSON line may claim:
per-launch DRAM traffic is reported only from a committed ncu capture of the
same kernel source, and the config object names how the norm and the rotary
write ran."""
import hashlib
import json
import os
import shutil
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _copy_tree(tmp_path, edit=None):
    """A minimal copy of the repository layout bench._traffic reads: the
    committed traffic file and the kernel sources it names."""
    entries = json.load(open(os.path.join(ROOT, "profiles", "ncu_traffic.json")))["entries"]
    os.makedirs(tmp_path / "profiles")
    for e in entries:
        dst = tmp_path / e["source"]
        os.makedirs(dst.parent, exist_ok=True)
        shutil.copy(os.path.join(ROOT, e["source"]), dst)
    if edit:
        edit(tmp_path, entries)
    json.dump({"entries": entries}, open(tmp_path / "profiles" / "ncu_traffic.json", "w"))
    return entries


def test_traffic_comes_from_a_capture_of_the_same_source(tmp_path, monkeypatch):
    entries = _copy_tree(tmp_path)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    for e in entries:
        src = open(tmp_path / e["source"], "rb").read()
        assert hashlib.sha256(src).hexdigest()[:16] == e["source_sha"], e["source"]
        assert bench._traffic(e["class"], e["workload"]) == e["bytes_per_launch"]
    assert bench._traffic("gemm", "no_such_workload") is None


def test_traffic_is_null_once_the_kernel_source_changed(tmp_path, monkeypatch):
    def touch_gemm(root, entries):
        p = root / "paper_2609_01338_gb300" / "csrc" / "gemm.cu"
        p.write_text(p.read_text() + "\n// changed\n")
    entries = _copy_tree(tmp_path, touch_gemm)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    for e in entries:
        got = bench._traffic(e["class"], e["workload"])
        if e["source"].endswith("gemm.cu"):
            assert got is None
        else:
            assert got == e["bytes_per_launch"]


def test_config_names_the_norm_and_rotary_paths():
    sc = {"model": {"n_layers": 2, "d_model": 256, "n_q_heads": 4, "n_kv_heads": 2, "head_dim": 64,
                    "ffn_dim": 688, "vocab": 1024, "kv_dtype": 0},
          "context": 512, "evict_tail": 256, "mode": "drop", "prompt": 32}
    base = bench._config("tiny", sc, "none", 1)
    assert base["rmsnorm"].startswith("folded") and base["rope_kv_write"] == "its own launch"
    abl = bench._config("tiny", sc, "none", 1, separate_norm=True, fused_rope=True)
    assert abl["rmsnorm"] == "separate launches"
    assert abl["rope_kv_write"].startswith("inside the QKV projection")
