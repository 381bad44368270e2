"""The NVFP4 block-scale code s_b = E4M3(fp32(t / 6)) (Sec. 4, two-level
NVFP4 scaling) is computed in the kernels without a division: the product
with RN(1/6) plus one fused correction step.  Its fp32 quotient may differ
from the correctly rounded one where that is subnormal, so the contract
checked here is the one the format needs: the E4M3 code equals the code of
the correctly rounded quotient for every fp32 t in [0, 4096] (exhaustively),
for sampled t above, for +inf, and NaN stays NaN."""
import os
import shutil
import subprocess

import pytest

from conftest import ROOT

pytestmark = pytest.mark.gpu


def test_block_scale_division_exhaustive(tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    exe = str(tmp_path / "div6")
    src = os.path.join(ROOT, "tests", "gpu_checks", "scale_div6_exhaustive.cu")
    inc = os.path.join(ROOT, "paper_2609_21849_gb300", "csrc")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                    "-I" + inc, "-I" + os.path.join(ROOT, "include"), src, "-o", exe],
                   check=True, capture_output=True, timeout=300)
    out = subprocess.run([exe], check=True, capture_output=True, text=True, timeout=120).stdout
    fields = out.split()
    assert fields[0] == "mismatches" and fields[1] == "0", out
    assert fields[3] == "1", out
