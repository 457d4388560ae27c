"""Host logic of bench.py's roofline.traffic: the committed one-launch DRAM record of the
small workload, keyed by the kernel source's SHA-256 and scaled by algorithmic bytes."""
import hashlib
import os

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _records():
    out = {}
    for ln in open(os.path.join(ROOT, "profiles", "dram_traffic_small.md")):
        if ln.startswith("traffic:"):
            kv = dict(x.split("=", 1) for x in ln[len("traffic:"):].split())
            out[kv["kernel"]] = kv
    return out


def test_committed_record_is_consistent_and_keyed_to_the_source():
    """Each record's read and write add up to per_launch. While its SHA-256 is that of the
    committed kernel source, the bench scales it by the launch's algorithmic bytes; once the
    source has changed, the bench reports no traffic until the record is taken again."""
    sha = hashlib.sha256(open(os.path.join(ROOT, "paper_2607_19058_gb300", "csrc", "skew_kernels.cu"), "rb").read()).hexdigest()
    recs = _records()
    assert {"k_apply_rows", "k_rowsq", "k_finalize"} <= set(recs)
    alg = 41_385_197_568
    for k, kv in recs.items():
        assert int(kv["read"]) + int(kv["write"]) == int(kv["per_launch"])
        if kv["source_sha256"] == sha:
            assert bench.recorded_traffic(k, alg) == round(int(kv["per_launch"]) * alg / int(kv["alg_bytes"]))
        else:
            assert bench.recorded_traffic(k, alg) is None


def _fake_root(tmp_path, source, record_lines):
    csrc = tmp_path / "paper_2607_19058_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (csrc / "skew_kernels.cu").write_bytes(source)
    prof = tmp_path / "profiles"
    prof.mkdir()
    (prof / "dram_traffic_small.md").write_text("\n".join(record_lines) + "\n")
    return str(tmp_path)


def test_a_changed_kernel_source_gives_no_traffic(tmp_path):
    src = b"// kernels\n"
    sha = hashlib.sha256(src).hexdigest()
    line = f"traffic: kernel=k_apply_rows workload=small read=6 write=4 per_launch=10 alg_bytes=5 source_sha256={sha}"
    root = _fake_root(tmp_path, src, [line])
    assert bench.recorded_traffic("k_apply_rows", 50, root=root) == 100     # 10 * 50 / 5
    assert bench.recorded_traffic("k_rowsq", 50, root=root) is None          # no record
    (tmp_path / "paper_2607_19058_gb300" / "csrc" / "skew_kernels.cu").write_bytes(b"// changed\n")
    assert bench.recorded_traffic("k_apply_rows", 50, root=root) is None     # stale record


def test_missing_record_file_gives_no_traffic(tmp_path):
    (tmp_path / "paper_2607_19058_gb300" / "csrc").mkdir(parents=True)
    (tmp_path / "paper_2607_19058_gb300" / "csrc" / "skew_kernels.cu").write_bytes(b"x")
    assert bench.recorded_traffic("k_apply_rows", 50, root=str(tmp_path)) is None
