"""bench.py's `roofline.traffic`: DRAM bytes from a committed ncu capture are reported
only while the kernel's sources (its .cu file and the headers it includes) are the
ones the capture was taken with; any change to one of them makes the field null."""

import importlib.util
import json
import os
import shutil

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _bench():
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def _tree(tmp_path):
    """A copy of the kernel sources and profiles/ under tmp_path, laid out like the repo."""
    csrc = tmp_path / "paper_2607_18171_gb300" / "csrc"
    csrc.mkdir(parents=True)
    for name in ("frt_attention.cu", "frt_ptx.cuh", "frt_internal.h"):
        shutil.copy(os.path.join(ROOT, "paper_2607_18171_gb300", "csrc", name), csrc / name)
    (tmp_path / "profiles").mkdir()
    return csrc


def test_committed_records_name_their_capture_and_sources():
    recs = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    assert recs, "no traffic records"
    for wl, rec in recs.items():
        assert rec["dram_bytes_per_launch"] > 0, wl
        assert len(rec["sources_sha256"]) == 64, wl
        assert os.path.exists(os.path.join(ROOT, rec["capture"])), (wl, rec["capture"])


def test_traffic_follows_every_kernel_source(tmp_path):
    b = _bench()
    csrc = _tree(tmp_path)
    b.ROOT = str(tmp_path)
    sha = b.kernel_sources_sha("frt_attention.cu")
    rec = {"stream720p": {"sources_sha256": sha, "dram_bytes_per_launch": 123}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    assert b.traffic_record("frt_attention.cu", "stream720p") == 123
    assert b.traffic_record("frt_attention.cu", "dit14b") is None
    # a change to the kernel file or to either header voids the record
    for name in ("frt_attention.cu", "frt_ptx.cuh", "frt_internal.h"):
        path = csrc / name
        original = path.read_bytes()
        path.write_bytes(original + b"\n// changed\n")
        assert b.traffic_record("frt_attention.cu", "stream720p") is None, name
        path.write_bytes(original)
        assert b.traffic_record("frt_attention.cu", "stream720p") == 123, name
