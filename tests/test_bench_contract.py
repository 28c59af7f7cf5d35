"""bench.py's command-line contract, checked on the CPU: the reference arm
(the oracle timed on the host cores) prints one JSON line with the keys the
benchmark contract names, prints it once under a two-rank launch, the
warm-up rule is enforced, and the CUDA arm fails loudly instead of falling
back to the CPU when no GPU is present."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
BENCH = os.path.join(ROOT, "bench.py")


def run(args, timeout=300):
    return subprocess.run([sys.executable, *args], cwd=ROOT, capture_output=True, text=True,
                          timeout=timeout)


def json_lines(stdout):
    return [json.loads(l) for l in stdout.splitlines() if l.startswith("{")]


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_reference_arm_prints_the_contract_line():
    r = run([BENCH, "--impl", "reference", "--workload", "C1", "--steps", "1", "--warmup", "3"])
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference"
    assert d["unit"] == "nodes/s" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 3
    assert d["ms_per_step"] > 0 and d["data"] == "synthetic"
    assert isinstance(d["config"]["workload"], str) and d["config"]["workload"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"]
    assert cb["unit"] == d["unit"] and cb["sample"]
    assert cb["host_cores"] == os.cpu_count()
    e2e = d["e2e"]
    assert e2e["value"] == d["value"] and e2e["unit"] == d["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_reference_arm_under_two_ranks_prints_once():
    r = run(["-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
             "--master-addr", "127.0.0.1", "--master-port", str(free_port()), BENCH,
             "--impl", "reference", "--workload", "C1", "--gpus", "2", "--steps", "1",
             "--warmup", "3"])
    assert r.returncode == 0, r.stderr[-2000:]
    lines = json_lines(r.stdout)
    assert len(lines) == 1 and lines[0]["impl"] == "reference" and lines[0]["n_gpus"] == 2


def test_fewer_than_three_warmup_steps_are_refused():
    r = run([BENCH, "--impl", "reference", "--workload", "C1", "--steps", "1", "--warmup", "2"])
    assert r.returncode != 0 and "warmup" in r.stderr
    assert not json_lines(r.stdout)


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the behaviour without a GPU")
def test_cuda_arm_fails_without_a_gpu():
    r = run([BENCH, "--workload", "C1", "--steps", "1", "--warmup", "3"])
    assert r.returncode != 0
    assert not json_lines(r.stdout)


def _profile_fields(path):
    fields = {}
    with open(path) as f:
        for line in f:
            if ":" in line:
                k, v = line.split(":", 1)
                fields[k.strip()] = v.strip()
    return fields


def test_kernel_profiles_name_their_command_sources_and_traffic():
    """Every committed per-kernel ncu summary gives the full command (ncu with
    --clock-control none after a plain run of the same command), the source
    files it was taken on with their hash, and the DRAM bytes per launch."""
    import glob
    paths = [p for p in glob.glob(os.path.join(ROOT, "profiles", "*.txt"))
             if "source_sha256_16" in _profile_fields(p)]
    assert len(paths) >= 20
    for p in paths:
        f = _profile_fields(p)
        cmd = f.get("command", "")
        assert "ncu" in cmd and "--clock-control none" in cmd, p
        assert cmd.split("&&")[0].strip().startswith("python bench.py"), p
        assert "source_file" in f or "source_files" in f, p
        assert float(f["dram_bytes_per_launch"].split(" ")[0]) > 0, p


def test_profile_traffic_needs_the_current_source(monkeypatch):
    """bench.py reports a summary's DRAM bytes only while the hash of the
    kernel sources it names is the one recorded in it."""
    sys.path.insert(0, ROOT)
    import bench
    name = "backward_step_C4.txt"
    f = _profile_fields(os.path.join(ROOT, "profiles", name))
    recorded = f["source_sha256_16"].split(" ")[0]
    files = ["backward.cu", "pack.cu", "spmm.cu", "ablation.cu"]
    monkeypatch.setattr(bench, "sources_hash", lambda fs: recorded)
    assert bench.profile_file_traffic(name, files) == float(f["dram_bytes_per_launch"].split(" ")[0])
    monkeypatch.setattr(bench, "sources_hash", lambda fs: "0" * 16)
    assert bench.profile_file_traffic(name, files) is None
    assert bench.profile_file_traffic("no_such_profile.txt", files) is None


def test_workload_cache_returns_the_same_arrays(monkeypatch, tmp_path):
    """With BIGCN_BENCH_CACHE set, the first build saves the workload and the
    second loads it: the arrays (values and dtypes) are those drawn afresh."""
    sys.path.insert(0, ROOT)
    import numpy as np
    import bench
    monkeypatch.delenv("BIGCN_BENCH_CACHE", raising=False)
    _, fresh = bench.build_workload("C1")
    monkeypatch.setenv("BIGCN_BENCH_CACHE", str(tmp_path))
    _, first = bench.build_workload("C1")
    assert len(list(tmp_path.iterdir())) == 1
    _, second = bench.build_workload("C1")
    for k in bench.WORKLOAD_ARRAYS:
        for got in (first[k], second[k]):
            assert got.dtype == fresh[k].dtype and np.array_equal(got, fresh[k]), k


def test_warm_l2_lines_are_for_workloads_that_fit_l2():
    """The 2-layer line adds a warm-L2 figure only where the forward's bytes
    fit the 129 MB L2: the Cora-, Citeseer- and PubMed-shaped workloads, not
    the Reddit-shaped one."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2010_07565_gb300 import inputs
    nnz = {"C1": 10556, "C2": 9228, "C3": 88648, "C4": 114600000}
    for name, fits in (("C1", True), ("C2", True), ("C3", True), ("C4", False)):
        w = inputs.get_workload(name)
        assert (bench.workload_bytes(w, nnz[name]) < bench.L2_BYTES) == fits, name


def test_roofline_work_matches_the_profile_summaries():
    """The algorithmic bytes bench.py divides by a kernel's time are the ones
    the committed ncu summaries state for the same kernel and workload, and
    the L2 gather ceiling is the measured entry for the next row size up."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2010_07565_gb300 import inputs
    cases = [("C4", 114600000, "L1.spmm+L2.pack_rows+L2.xnor_gemm",
              "L1.spmm_L2.pack_rows_L2.xnor_gemm_C4.txt"),
             ("C4", 114600000, "L2.spmm", "L2.spmm_C4.txt"),
             ("C2", 9356, "L1.pack_rows+L1.xnor_gemm", "L1.pack_rows_L1.xnor_gemm_C2.txt")]
    for name, nnz, kernel, fname in cases:
        f = _profile_fields(os.path.join(ROOT, "profiles", fname))
        stated = float(f["algorithmic_bytes_per_launch"].split(" ")[0])
        work, unit, bound = bench.kernel_work(inputs.get_workload(name), nnz, kernel)
        assert (unit, bound) == ("bytes", "hbm") and work == stated, (name, kernel, work, stated)
    assert bench.l2_gather_peak(260) == (bench.L2_GATHER_GBS[512], 512)
    assert bench.l2_gather_peak(100) == (bench.L2_GATHER_GBS[128], 128)
    assert bench.l2_gather_peak(4096) == (bench.L2_GATHER_GBS[512], 512)
