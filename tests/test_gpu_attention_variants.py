"""The alternative attention kernels for head_dim 128 with 8 kv heads, checked with the same cases as the default
ones: the per-row decode-attention kernels (which the streaming kernel replaces; SR_ATTN_STREAM=0) and the
tcgen05 prefix pass and prefill attention (opt-in, measured slower than the mma.sync kernels; SR_PREFIX_TC=1,
SR_PREFILL_TC=1).  The switches are read once per process, so each set runs in a child."""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("env", [{"SR_ATTN_STREAM": "0"}, {"SR_PREFIX_TC": "1", "SR_PREFILL_TC": "1"}])
def test_alternative_attention_kernels(env):
    child = dict(os.environ, **env)
    r = subprocess.run([sys.executable, "-m", "pytest", "-q", "-x", "-m", "gpu", "-k", "decode_attention or prefill_attention",
                        "-p", "no:cacheprovider", os.path.join(ROOT, "tests", "test_gpu_kernels.py")], cwd=ROOT,
                       env=child, capture_output=True, text=True, timeout=900)
    assert r.returncode == 0, r.stdout[-4000:] + r.stderr[-2000:]
    assert " passed" in r.stdout
