"""The GPU's Box-Muller transform (zo_device.cuh: box_muller, sqrt(-2 ln ua) times
(cos, sin) of 2 pi ub in fp32) over every uniform the counter contract produces,
u = j 2^-24, j = 1 .. 2^24, against double precision: a probe built with nvcc from the
same header sweeps the radius with ub = 1 (cos = 1, sin = 0 exactly) and the angle at the
largest radius (ua = 2^-24).  A normal's error is at most the radius error plus the radius
times the angle error plus the product's rounding, and the sweep at the largest radius
bounds the angle error up to one more radius error and rounding; so every normal the
kernels can draw stays within 2 e_radius + e_sweep + 2^-21, which must be within the
normals' tolerance against the oracle."""
import os
import shutil
import subprocess

import pytest

from parity import NORMAL_ABS

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_box_muller_over_every_uniform(gpu, tmp_path):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    exe = str(tmp_path / "probe")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O3", "-std=c++17",
                    "-I", os.path.join(ROOT, "paper_2608_15665_gb300", "csrc"),
                    os.path.join(ROOT, "tests", "harness", "box_muller_probe.cu"), "-o", exe],
                   check=True, capture_output=True, text=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    vals = {line.split()[0]: float(line.split()[1]) for line in out.splitlines()}
    print("\n" + out)
    # any pair (ua, ub): |dz| <= e_rad(ua) + r_max |d cos(ub)| + half an ulp of z, and the
    # sweep gives r_max |d cos| <= e_sweep + e_rad(2^-24) + half an ulp (ulp at 5.77: 2^-21)
    bound = 2 * vals["radius"] + max(vals["zcos"], vals["zsin"]) + 2.0 ** -21
    assert bound <= NORMAL_ABS, (bound, out)
