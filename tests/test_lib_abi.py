"""The C-ABI library builds, loads and exports every entry point include/sr.h declares (CPU only)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2410_20290_gb300", "libsr.so")


@pytest.fixture(scope="module")
def lib_path():
    if not os.path.exists(LIB):
        from paper_2410_20290_gb300 import build
        build.build()
    return LIB


def test_exports_every_declared_symbol(lib_path):
    header = open(os.path.join(ROOT, "include", "sr.h")).read()
    declared = set(re.findall(r"\b(sr_[a-z_0-9]+)\s*\(", header))
    assert {"sr_init", "sr_generate", "sr_decode_step", "sr_score_partial", "sr_reject_compact"} <= declared
    lib = ctypes.CDLL(lib_path)
    missing = [s for s in sorted(declared) if not hasattr(lib, s)]
    assert not missing, missing
    nm = subprocess.run(["nm", "-D", "--defined-only", lib_path], capture_output=True, text=True).stdout
    exported = set(re.findall(r" T (sr_[a-z_0-9]+)$", nm, re.M))
    assert declared <= exported


def test_binding_names_match_header(lib_path):
    from paper_2410_20290_gb300 import binding
    for name in binding.declared_symbols():
        if name == "sr_last_error":
            continue
        assert hasattr(binding, name), name


def test_errors_without_device(lib_path):
    """Argument checks run before any device work and report through sr_last_error."""
    from paper_2410_20290_gb300 import binding as b
    import sr_inputs as si
    m = si.WORKLOADS["tiny"].gen
    with pytest.raises(b.SrError) as e:
        b.sr_init(m, None, m.replace(has_lm_head=0, has_scalar_head=1), None)
    assert e.value.status == b.SR_ERR_INVALID_ARG
    import numpy as np
    x = np.zeros(4, np.float32)
    with pytest.raises(b.SrError) as e:
        b.sr_init(m.replace(n_heads=3, n_kv_heads=2), x, m.replace(has_lm_head=0, has_scalar_head=1), x)
    assert e.value.status in (b.SR_ERR_UNSUPPORTED, b.SR_ERR_INVALID_ARG)


def test_host_only_entry_points_validate_arguments(lib_path):
    """Calls that do no device work check their arguments on the host: null contexts and impossible sizes."""
    from paper_2410_20290_gb300 import binding as b
    import sr_inputs as si
    m = si.WORKLOADS["llama8b_n1024"].gen
    for kind in (b.SR_REWARD_MODEL, b.SR_REWARD_LOGPROB):
        with pytest.raises(b.SrError) as e:
            b.sr_set_reward(None, kind)
        assert e.value.status == b.SR_ERR_INVALID_ARG
    with pytest.raises(b.SrError) as e:
        b.sr_set_profiling(None, 8)
    assert e.value.status == b.SR_ERR_INVALID_ARG
    for P, tau, n_max in ((0, 8, 16), (16, 0, 16), (16, 8, 0)):
        with pytest.raises(b.SrError) as e:
            b.sr_auto_b_init(m, 60 * 10 ** 9, P, tau, n_max)
        assert e.value.status == b.SR_ERR_INVALID_ARG
    assert b.sr_auto_b_init(m, 1000, 16, 8, 16) == 0          # a pool below one page: nothing fits (SR_ERR_OOM)
    assert "tau_min" in b.LIB.sr_last_error().decode()


def test_kernel_entry_points_reject_bad_arguments_on_the_host(lib_path):
    """The kernel-level calls check pointers, dtypes and epilogue codes before any device work, so a caller's
    mistake is an SR_ERR_INVALID_ARG status (with a message), never a launch on bad arguments.  The host arrays
    passed here are never dereferenced: every call returns at its argument check."""
    import numpy as np
    from paper_2410_20290_gb300 import binding as b
    import sr_inputs as si
    x = np.zeros(64, np.float32)
    ids = np.zeros(4, np.int32)
    cases = [
        lambda: b.sr_k_lm_head_sample(si.DT_F16, None, x, 4, 64, 16, ids, ids, 1, 1.0, 0.0, 0, ids),
        lambda: b.sr_k_lm_head_sample(si.DT_F32, x, x, 4, 64, 16, ids, ids, 1, 1.0, 0.0, 0, ids),   # 16-bit only
        lambda: b.sr_k_sample(None, 64, 4, 64, ids, ids, 1, 1.0, 0.0, 0, ids),
        lambda: b.sr_k_gemm(si.DT_F16, None, x, x, 4, 64, 16, 0),
        lambda: b.sr_k_gemm(si.DT_F16, x, x, x, 4, 64, 16, 9),                                     # no epilogue 9
        lambda: b.sr_k_decode_attention(si.DT_F16, None, x, ids, 1, ids, ids, 4, 32, 8, 128, 0, x),
    ]
    for call in cases:
        with pytest.raises(b.SrError) as e:
            call()
        assert e.value.status == b.SR_ERR_INVALID_ARG
        assert b.LIB.sr_last_error().decode()
