"""The tcgen05 GEMM's alternative tile shapes, checked with the same GEMM cases as the default launch.

The launcher reads its tile overrides (SR_GEMM_SKINNY=0 / 1: never / always the transposed split-K kernel for M <= 512;
SR_GEMM_PAIR: 256 x 256 tiles computed by a CTA pair with
cta_group::2 MMAs; SR_GEMM_TM: 256-row tiles with two MMAs per W tile on one SM; SR_GEMM_BN: the N-tile
width of the 128-row tiles; SR_GEMM_STREAMK=1: stream-K shares of k-blocks on 128 x 256 tiles) once
per process, so each variant
runs the GEMM cases of test_gpu_kernels.py in a child process of its own.
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("env", [{"SR_GEMM_SKINNY": "0"}, {"SR_GEMM_SKINNY": "1"}, {"SR_GEMM_PAIR": "1"},
                                 {"SR_GEMM_TM": "256"}, {"SR_GEMM_BN": "64"}, {"SR_GEMM_BN": "128"},
                                 {"SR_GEMM_BN": "192"},
                                 {"SR_GEMM_STREAMK": "1"}])
def test_gemm_tile_variant(env):
    child = dict(os.environ, **env)
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-k", "gemm_tc", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_gpu_kernels.py")], cwd=ROOT, env=child,
                       capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout and "skipped" not in r.stdout.split("\n")[-2]
