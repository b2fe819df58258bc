"""Host-side helpers of bench.py (no GPU): the key that ties the committed
DRAM counters to the attention kernel's code."""
import importlib.util
import json
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_code_hash_ignores_comments_not_code(tmp_path):
    b = _bench()
    base = "int f(int x) {\n  return x + 1;  // one more\n}\n"
    p = tmp_path / "k.cu"
    p.write_text(base)
    h0 = b.code_sha256(str(p))
    p.write_text("/* header\n   comment */\n" + base.replace("// one more", "// a different note") + "\n\n")
    assert b.code_sha256(str(p)) == h0
    p.write_text(base.replace("x + 1", "x + 2"))
    assert b.code_sha256(str(p)) != h0


def test_traffic_record_shape_and_lookup(tmp_path, monkeypatch):
    b = _bench()
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))["tree_attn_tc_kernel"]
    assert rec["dram_bytes_per_launch"] == rec["dram_read_bytes"] + rec["dram_write_bytes"]
    assert len(rec["code_sha256"]) == 64 and rec["workload"] == "batched"
    # a workload other than the captured one, or a changed kernel, reports no traffic
    assert b.measured_traffic("tree_attn_tc_kernel", "tiny") is None
    # the same source under another root: the recorded key finds the bytes, a
    # wrong key finds none
    src = tmp_path / rec["source"]
    src.parent.mkdir(parents=True)
    src.write_text(open(os.path.join(ROOT, rec["source"])).read())
    fake = tmp_path / "profiles"
    fake.mkdir()
    monkeypatch.setattr(b, "ROOT", str(tmp_path))
    right = dict(rec, code_sha256=b.code_sha256(str(src)))
    (fake / "traffic.json").write_text(json.dumps({"tree_attn_tc_kernel": right}))
    assert b.measured_traffic("tree_attn_tc_kernel", "batched") == rec["dram_bytes_per_launch"]
    (fake / "traffic.json").write_text(json.dumps({"tree_attn_tc_kernel": dict(rec, code_sha256="0" * 64)}))
    assert b.measured_traffic("tree_attn_tc_kernel", "batched") is None
