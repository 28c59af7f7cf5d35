"""The measurement behind the choice of instruction for the XNOR product:
builds and runs tests/probes/instruction_rates.cu on the GPU (b1 tensor-core
MMA against CUDA-core POPC), checks the probe's own fragment-layout check and
prints the rates (-s shows them)."""
import os
import re
import shutil
import subprocess
import tempfile

import pytest

pytestmark = pytest.mark.gpu
PROBE = os.path.join(os.path.dirname(__file__), "probes", "instruction_rates.cu")


def test_instruction_rates(cuda_device):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "rates")
        subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-o", exe,
                        PROBE], check=True)
        out = subprocess.run([exe], check=True, capture_output=True, text=True, timeout=120).stdout
    print(out)
    assert out.count("0 mismatches of 128") == 2
    popc = float(re.search(r"popc32: [\d.]+ ms, [\d.]+ T popc/s = ([\d.]+) T bit-ops/s", out).group(1))
    assert popc > 0.0
