"""A measurement, not a parity test: builds and runs tests/probes/l2_gather.cu
on the GPU -- random row gathers (16 to 512-byte rows) from L2-resident and
HBM-resident buffers with plain loads and with cp.async, cp.async into staged
rows of a padded or XOR-swizzled pitch, and the rate of the
f16 mma.sync the tensor-core aggregation issues -- and prints the rates
(-s shows them). These are the ceilings the aggregation kernels are reported
against; the test only checks that the probe ran and produced rates."""
import os
import re
import shutil
import subprocess
import tempfile

import pytest

pytestmark = pytest.mark.gpu
PROBE = os.path.join(os.path.dirname(__file__), "probes", "l2_gather.cu")


def test_gather_rates(cuda_device):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    with tempfile.TemporaryDirectory() as d:
        exe = os.path.join(d, "gather")
        subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-o", exe,
                        PROBE], check=True)
        out = subprocess.run([exe], check=True, capture_output=True, text=True,
                             timeout=300).stdout
    print(out)
    rates = [float(x) for x in re.findall(r"gathered\s+([\d.]+) GB/s", out)]
    assert len(rates) == 41 and min(rates) > 0.0
    assert re.search(r"mma.sync m16n8k16 f16 -> f32: .* ([\d.]+) TFLOP/s", out)
