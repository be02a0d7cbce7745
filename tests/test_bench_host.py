"""Host-side plumbing of bench.py that needs no GPU."""
import hashlib
import importlib.util
import os

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_traffic_is_reported_only_for_the_profiled_sources(tmp_path, monkeypatch):
    bench = _bench()
    csrc = tmp_path / "paper_2609_32046_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    for f in bench.KERNEL_SOURCES:
        (csrc / f).write_bytes(("// " + f + "\n").encode())
    h = hashlib.sha256()
    for f in bench.KERNEL_SOURCES:
        h.update((csrc / f).read_bytes())
    (tmp_path / "profiles" / "k_demo_wl.md").write_text(
        "# demo\n\nsource_sha256: %s\ntraffic_bytes_per_launch: 123456\n" % h.hexdigest())
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_for("k_demo", "wl") == 123456
    assert bench.traffic_for("k_demo", "other") is None          # no summary for that workload
    (csrc / bench.KERNEL_SOURCES[-1]).write_bytes(b"// edited\n")  # the kernel changed since the capture
    assert bench.traffic_for("k_demo", "wl") is None


def test_committed_summaries_name_a_full_hash_and_a_byte_count():
    bench = _bench()
    import re
    found = 0
    for name in os.listdir(os.path.join(ROOT, "profiles")):
        text = open(os.path.join(ROOT, "profiles", name)).read()
        if "source_sha256" not in text:
            continue
        found += 1
        assert re.search(r"source_sha256:\s*[0-9a-f]{64}\b", text), name
        assert re.search(r"traffic_bytes_per_launch:\s*[0-9]+\b", text), name
    assert found >= 2
    assert bench.KERNEL_SOURCES == ("cb_score_tc.cu", "cb_sm100.cuh", "cb_internal.cuh")
