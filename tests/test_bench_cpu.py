"""Host logic of bench.py, without a GPU: the committed ncu figures are kept
only while their kernel's source is unchanged, the whole-job aggregate, the
workload config shared by both arms, and the reference arm's JSON line."""
import hashlib
import json

import pytest

import bench


def test_ncu_figures_follow_the_kernel_source(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_2607_14431_gb300" / "csrc"
    csrc.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    src = csrc / "k.cu"
    src.write_text("__global__ void k() {}\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text(
        "# comment\n"
        f"kernel=k source=k.cu sha={sha} bytes_per_launch=1234 alu_inst_per_compression=952\n"
        "kernel=gone source=missing.cu sha=0123456789abcdef bytes_per_launch=5\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.load_traffic() == {"k": 1234.0}
    assert bench.sha_alu_ops_per_compression("k") == 952.0
    src.write_text("__global__ void k() { /* changed */ }\n")
    assert bench.load_traffic() == {} and bench.sha_alu_ops_per_compression("k") is None


def test_aggregate_on_one_rank():
    ms, gbs = bench.aggregate(59.6, 10, 38_650_000_000, 1, None)
    assert ms == pytest.approx(5.96)
    assert gbs == pytest.approx(38.65e9 / 5.96e-3 / 1e9)


def test_config_names_the_workload_and_replicas():
    c = bench.config_12b(world=4)
    assert c["seq_len"] == 32768 and c["global_batch"] == 4 and c["parallelism"] == "replicas4"
    assert c["workload"].startswith("12b-single-graft: L48 Hq16/Hkv8 D256 P64")
    assert "larger than L2" in c["l2"]


def test_reference_arm_line(monkeypatch):
    monkeypatch.setattr(bench, "oracle_sample", lambda layers: (0.5, 2_000_000_000, 16))

    class A:
        gpus, steps, warmup = 1, 3, 1
    line = bench.run_reference(A())
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["value"] == pytest.approx(4.0) and line["unit"] == "GB/s"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == 16
    assert line["e2e"] == {"value": line["value"], "unit": "GB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    json.dumps(line)
