"""bench.py's JSON contract on the CPU: the reference arm (the oracle timed on the host cores)
prints one line with the fields its consumers parse, and under torchrun only rank 0 prints."""
import json
import os
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(cmd, timeout=600):
    env = dict(os.environ, MASTER_ADDR="127.0.0.1")
    p = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=timeout)
    assert p.returncode == 0, p.stderr[-2000:]
    return [l for l in p.stdout.splitlines() if l.startswith("{")]


def _check_line(d, n_gpus):
    sys.path.insert(0, ROOT)
    import bench
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["n_gpus"] == n_gpus and d["steps"] >= 1 and d["scaling"] == "weak"
    assert d["data"] == "synthetic" and d["vs_baseline"] is None
    assert d["config"]["workload"] and "model" not in d["config"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["sample"]
    assert cb["value"] == d["value"] and cb["unit"] == d["unit"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["unit"] == d["unit"]
    assert e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_prints_one_contract_line():
    lines = _run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1",
                  "--warmup", "0"])
    assert len(lines) == 1
    _check_line(json.loads(lines[0]), 1)


def _free_port():
    import socket
    with socket.socket() as sk:
        sk.bind(("127.0.0.1", 0))
        return sk.getsockname()[1]


def test_reference_arm_under_torchrun_prints_on_rank_0_only():
    pytest.importorskip("torch.distributed.run")
    lines = _run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
                  "--nproc-per-node=2", "--master-addr", "127.0.0.1",
                  "--master-port", str(_free_port()),
                  "bench.py", "--impl", "reference", "--gpus", "2", "--steps", "1",
                  "--warmup", "0"])
    assert len(lines) == 1
    _check_line(json.loads(lines[0]), 2)


def test_reference_arm_launches_its_own_ranks_for_gpus_2():
    """--gpus 2 without torchrun's environment starts two ranks itself; only rank 0 prints."""
    pytest.importorskip("torch.distributed.run")
    env = {k: v for k, v in os.environ.items()
           if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    p = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    _check_line(json.loads(lines[0]), 2)


def test_rank_count_must_match_gpus():
    env = dict(os.environ, RANK="0", LOCAL_RANK="0", WORLD_SIZE="1")
    p = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], cwd=ROOT, env=env,
                       capture_output=True, text=True, timeout=300)
    assert p.returncode != 0 and "--gpus 2" in p.stderr
    assert not [l for l in p.stdout.splitlines() if l.startswith("{")]


def test_launcher_reaches_process_group_with_two_ranks():
    """The launcher the main arm uses for --gpus 2, with gloo standing in for NCCL: both
    ranks join one process group of size 2 through bench.init_dist and gather timings."""
    pytest.importorskip("torch.distributed.run")
    probe = os.path.join(ROOT, "tests", "bench_rank_probe.py")
    code = ("import sys; sys.path.insert(0, %r); import bench; "
            "sys.exit(bench.launch_ranks(2, [], script=%r))" % (ROOT, probe))
    env = {k: v for k, v in os.environ.items()
           if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    p = subprocess.run([sys.executable, "-c", code], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=300)
    assert p.returncode == 0, p.stderr[-2000:]
    lines = [l for l in p.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["world"] == 2 and d["backend"] == "gloo" and d["times"] == [0.5, 0.75]
    assert d["value"] == pytest.approx(64 * 100 * 2 / 0.75)


@pytest.mark.gpu
def test_main_arm_prints_one_contract_line():
    lines = _run([sys.executable, "bench.py", "--steps", "8", "--warmup", "4",
                  "--config-steps", "32", "--config-cpu-s", "0.2",
                  "--full-seq-max-steps", "3", "--cpu-budget-s", "1"])
    assert len(lines) == 1
    d = json.loads(lines[0])
    sys.path.insert(0, ROOT)
    import bench
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT and "impl" not in d
    assert d["value"] > 0 and d["n_gpus"] == 1 and d["warmup"] >= 3
    assert d["steps"] >= 1000 and d["config"]["steps_requested"] == 8  # the 1000-step floor
    assert d["config"]["step_us_distribution"]["replays"] >= 100
    r = d["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] > 0
    assert 0 < r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["traffic"] is None or r["traffic"] > 0
    assert d["gpu_launches"] == 2 * d["steps"]
    assert d["clocks"]["sm_max_mhz"] > 0 and d["clocks"]["samples_in_timed_region"] >= 3
    pc = d["per_config"]
    for name in ("single_block_b1_l32_bf16", "mixed_mask_b8_l32_bf16",
                 "tie_groups_b16_l64_fp32"):
        for r in pc[name]["rules"].values():
            assert r["us_per_step"] > 0 and r["selections_per_s"] > 0
            assert 0 < r["frac_of_measured_hbm"] < 2
        assert pc[name]["cpu_baseline"]["kind"] == "oracle"
    assert len(pc["mixed_mask_b8_l32_bf16"]["rules"]) == 7
    assert pc["tie_groups_b16_l64_fp32"]["identical_decisions_profile_factor"] is True
    fs = pc["full_seq_b16_l1024_fp32"]
    assert fs["profile f=1"]["steps"] == 3 and fs["factor f=1"]["per_step_ms_median"] > 0
    rb = pc["serving_b64_l32_bf16_robust"]
    assert rb["robust_us_per_step"] > 0 and rb["profile_us_per_step"] > 0
    dl = d["decode_loop"]
    assert dl["identical_decisions"] is True and dl["steps"] == sum(dl["nfe_per_block"])
    assert dl["device_loop"]["tokens_per_s"] > 0
    for b in ("B=64", "B=32", "B=16", "B=1"):
        lm = d["lmhead"][b]
        assert lm["fused_ms"] > 0 and 0 < lm["frac_of_burst_bf16"] < 1.3
    ev = d["evolving"]  # the serving workload with masks evolving until every row finishes
    assert ev["us_per_step"] > 0 and ev["period_steps"] == len(ev["masked_rows_per_step"])
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] > 0 and e["d2h_bytes_per_step"] > 0
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] > 0 and cb["sample"]


def test_ncu_traffic_only_for_its_workload_and_sources(monkeypatch, tmp_path):
    """The roofline's `traffic` comes from the committed ncu summary of the serving workload
    only while the reduction's sources hash to the value recorded there (a kernel changed
    since the capture reads as null), and never for another workload."""
    sys.path.insert(0, ROOT)
    import bench
    t = bench.ncu_traffic("serving_b64_l32_bf16")
    assert t is not None and t > 0, "profile summary is stale: re-capture it on these sources"
    assert bench.ncu_traffic("single_block_b1_l32_bf16") is None
    changed = tmp_path / "vocab_reduce.cu"
    changed.write_text("// another kernel\n")
    monkeypatch.setattr(bench, "KERNEL_SOURCES", [str(changed)])
    assert bench.ncu_traffic("serving_b64_l32_bf16") is None
