"""Host-side checks of the C ABI (no GPU needed): the library builds, loads
and exports every entry point include/simsd.h declares, and host argument
validation rejects bad calls before any CUDA work.  Also checks that the
product package never imports the oracle."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2606_02544_gb300 import build, simsd
    build.build()
    return simsd.load_library()


def _declared():
    with open(os.path.join(ROOT, "include", "simsd.h")) as f:
        text = f.read()
    return re.findall(r"SIMSD_API\s+[\w\s\*]+?\b(simsd_\w+)\s*\(", text)


def test_header_declares_the_boundary():
    names = set(_declared())
    assert {"simsd_build_mask", "simsd_verify_attention", "simsd_accept", "simsd_kv_commit"} <= names


def test_every_declared_symbol_is_exported(lib):
    from paper_2606_02544_gb300 import simsd
    for name in _declared():
        assert hasattr(lib, name), name
    assert set(_declared()) == set(simsd.EXPORTED)


def test_host_validation_without_gpu(lib):
    assert lib.simsd_version() == 10100
    P = ctypes.c_void_p
    one = ctypes.c_void_p(16)
    # gamma outside [1, 32]
    assert lib.simsd_build_mask(None, one, 1, 0, one, one, one, None, None, None) == 1
    assert lib.simsd_build_mask(None, one, 1, 33, one, one, one, None, None, None) == 1
    F = ctypes.c_float
    # rope_pos given without a positive, finite rope_theta
    for theta in (0.0, -1.0, float("inf"), float("nan")):
        rc = lib.simsd_verify_attention(1, one, one, one, one, one, 4, one, 1, 64, one, one, one, one, F(theta), 1, 4,
                                        8, 8, 128, F(0.0), one, None, 0, None, None)
        assert rc == 1
        rc = lib.simsd_kv_commit(1, one, one, 1, one, one, one, F(theta), one, one, one, 4, one, 1, 64, one, 1, 4,
                                 8, 128, None, None)
        assert rc == 1
    # Hq not a multiple of Hkv
    rc = lib.simsd_verify_attention(1, one, one, one, one, one, 4, one, 1, 64, one, one, one, None, F(0.0), 1, 4, 6,
                                    4, 128, F(0.0), one, None, 0, None, None)
    assert rc == 1
    # vocab out of range
    assert lib.simsd_accept(one, one, 1, 4, 0, one, one, None, None, None) == 1
    # stochastic acceptance: temperature must be positive and finite, gamma in [1, 32]
    for t, g, v in ((0.0, 4, 10), (-1.0, 4, 10), (float("inf"), 4, 10), (float("nan"), 4, 10), (1.0, 0, 10),
                    (1.0, 33, 10), (1.0, 4, 0)):
        assert lib.simsd_accept_sampled(one, one, one, one, one, F(t), 1, g, v, one, one, None, None) == 1
    assert lib.simsd_accept_sampled(one, None, one, one, one, F(1.0), 1, 4, 10, one, one, None, None) == 1
    assert lib.simsd_accept_sampled(None, None, None, None, None, F(1.0), 0, 4, 10, None, None, None, None) == 0
    # empty batches are no-ops that touch nothing
    assert lib.simsd_accept(None, None, 0, 4, 10, None, None, None, None, None) == 0
    # the wait-expiry test hook validates its arguments on the host
    assert lib.simsd_debug_expire_next_wait(0, 200) == 1
    assert lib.simsd_debug_expire_next_wait(3, 200) == 1
    assert lib.simsd_debug_expire_next_wait(1, 5) == 1
    assert lib.simsd_debug_expire_next_wait(2, 2000000) == 1
    assert lib.simsd_check_error(None, None, None) == 1
    assert b"null error word" in lib.simsd_last_error()


def test_product_never_imports_the_oracle():
    pkg = os.path.join(ROOT, "paper_2606_02544_gb300")
    for dirpath, _, files in os.walk(pkg):
        for fn in files:
            if fn.endswith((".py", ".cu", ".cuh", ".h")):
                with open(os.path.join(dirpath, fn)) as f:
                    src = f.read()
                assert "simsd_oracle" not in src and "import oracle" not in src and "from oracle" not in src, fn
