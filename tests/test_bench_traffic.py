"""The committed DRAM-traffic summary that bench.py attaches to each
workload's roofline kernel: every entry names a benchmarked workload, a
kernel source file of the package and a positive byte count, and the lookup
returns it only while that source's hash matches (a changed kernel reports
no traffic rather than a stale one)."""
import hashlib
import os
import sys

ROOT = os.path.join(os.path.dirname(__file__), "..")
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def entries():
    out = []
    for line in open(os.path.join(ROOT, "profiles", "ncu_traffic.txt")):
        if line.startswith("#") or not line.strip():
            continue
        out.append(line.split())
    return out


def test_every_entry_is_well_formed():
    e = entries()
    assert e
    for f in e:
        assert len(f) == 4, f
        assert f[0] in (bench.WORKLOAD,) + tuple(bench.OTHER_WORKLOADS), f
        src = os.path.join(ROOT, "paper_2504_13850_gb300", "csrc", f[2].split(":")[0])
        assert os.path.exists(src), f
        assert len(f[2].split(":")[1]) == 12 and float(f[3]) > 0, f


def test_lookup_follows_the_source_hash(tmp_path, monkeypatch):
    src = tmp_path / "paper_2504_13850_gb300" / "csrc"
    src.mkdir(parents=True)
    (src / "k.cu").write_text("kernel v1")
    h = hashlib.sha1(b"kernel v1").hexdigest()[:12]
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text(f"# comment\nvgg tc_conv_wgrad k.cu:{h} 123\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_for("tc_conv_wgrad", "vgg") == 123.0
    assert bench.traffic_for("tc_conv_wgrad", "resnet") is None
    (src / "k.cu").write_text("kernel v2")
    assert bench.traffic_for("tc_conv_wgrad", "vgg") is None
