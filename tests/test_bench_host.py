"""Host logic of bench.py on CPU: the per-step DRAM traffic ingest, the
workload variants and the reference arm's JSON line."""
import argparse
import json
import os
import subprocess
import sys

import pytest

import bench
from paper_2505_00315_gb300 import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _csv_row(i, name, metric, unit, value):
    # the column layout of ncu --csv --metrics output
    return (f'"{i}","1","python3.12","127.0.0.1","{name}","1","7","(256, 1, 1)","(128, 1, 1)",'
            f'"0","10.3","Command line profiler metrics","{metric}","{unit}","{value}"\n')


def test_ingest_counts_traffic_per_step(tmp_path, monkeypatch):
    # two steps; attn_bwd launches two kernels a step (the large-k backward
    # and its dQ split), w_bwd one: bytes are summed per stage and divided by
    # the steps, counted from the TopK launches
    head = ('"ID","Process ID","Process Name","Host Name","Kernel Name","Context","Stream",'
            '"Block Size","Grid Size","Device","CC","Section Name","Metric Name","Metric Unit",'
            '"Metric Value"\n')
    rows, i = [], 0
    for _ in range(2):
        for name, mb in (("mosa::topk_select_kernel(const float *)", 0.5),
                         ("mosa::attn_bwd_tc_kernel(BwdParams)", 40.0),
                         ("mosa::dq_finish_kernel(const float *)", 8.0),
                         ("void mosa::tc_gemm_kernel<4>(TcParams)", 30.0)):
            rows.append(_csv_row(i, name, "dram__bytes_read.sum", "Mbyte", mb))
            rows.append(_csv_row(i, name, "dram__bytes_write.sum", "byte", 0))
            rows.append(_csv_row(i, name, "gpu__time_duration.sum", "usecond", 1.0))
            i += 1
    csv = tmp_path / "dram.csv"
    csv.write_text("==PROF== banner line\n" + head + "".join(rows))
    profiles = tmp_path / "profiles"
    profiles.mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "source_digest", lambda: "digest")
    bench.ingest_ncu(str(csv), "wl")
    ent = json.load(open(profiles / "traffic.json"))["wl"]
    assert ent["attn_bwd"]["bytes_per_step"] == pytest.approx(48e6)
    assert ent["attn_bwd"]["launches"] == 4 and ent["attn_bwd"]["steps"] == 2
    assert ent["w_bwd"]["bytes_per_step"] == pytest.approx(30e6)
    assert bench.traffic_for("w_bwd", "wl") == pytest.approx(30e6)
    monkeypatch.setattr(bench, "source_digest", lambda: "other sources")
    assert bench.traffic_for("w_bwd", "wl") is None


def test_variant_names_and_config():
    base = W.CONFIGS[W.BENCH_CONFIG]
    a = argparse.Namespace(rope=True, first_token=False, dense_heads=4, window=512)
    cfg = bench.variant(base, a)
    assert cfg.name == base.name + "+rope+dense4w512" and cfg.rope and not cfg.first_token
    blk = bench.config_block(cfg, a)
    assert blk["H_dense"] == 4 and blk["window"] == 512 and blk["rope"] is True
    plain = argparse.Namespace(rope=False, first_token=False, dense_heads=0, window=0)
    assert bench.variant(base, plain).name == base.name
    assert "H_dense" not in bench.config_block(base, plain)


def test_reference_arm_prints_one_line():
    # the oracle as the reference arm, one short step
    # (a small workload: one sequence of the default one takes the oracle ~20 s)
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--config", "B8_T1024_d512_H16_k128", "--steps", "1", "--warmup", "0"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["value"] > 0 and j["unit"] == "tokens/s"
    assert j["config"]["workload"] == "B8_T1024_d512_H16_k128"
    assert j["cpu_baseline"]["kind"] == "oracle"
    assert j["e2e"]["h2d_bytes_per_step"] == 0
