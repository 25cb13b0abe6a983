"""The checked build (libjab_checked.so, nvcc -DJAB_CHECKED=1): bounds checks before the kernels'
computed global accesses report JAB_ERR_DEVICE_ASSERT and skip the access instead of faulting.

The library is chosen when the binding first loads (JAB_CHECKED=1 in the environment), so the checked
runs happen in child processes: the self-test of the mechanism, and parity cases of every kernel
family run on the checked library, which must raise no check (device status 0 after each case).
"""
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _child(code_or_args, timeout=900):
    env = dict(os.environ, JAB_CHECKED="1")
    args = [sys.executable, "-c", code_or_args] if isinstance(code_or_args, str) else code_or_args
    return subprocess.run(args, cwd=ROOT, env=env, capture_output=True, text=True, timeout=timeout)


@pytest.fixture(scope="module", autouse=True)
def _checked_library():
    from paper_2609_34866_gb300 import build
    build.build(checked=True)


def test_bounds_check_self_test_skips_the_access_and_raises_the_status():
    r = _child(
        "import torch, paper_2609_34866_gb300 as J\n"
        "assert J.lib_path().endswith('libjab_checked.so')\n"
        "n = 200\n"
        "buf = torch.full((n + 1,), -7, dtype=torch.int32, device='cuda')\n"
        "assert J.jab_selftest_bounds_check(buf, n) == 0\n"
        "st = J.jab_get_device_status()\n"
        "b = buf.cpu()\n"
        "assert st == 9, st\n"
        "assert b[n].item() == -7 and torch.equal(b[:n], torch.arange(n, dtype=torch.int32))\n"
        "assert J.jab_get_device_status() == 0\n"
        "print('ok')\n")
    assert r.returncode == 0 and "ok" in r.stdout, r.stdout + r.stderr


def test_normal_build_has_no_bounds_checks():
    import torch
    from tests.harness import J
    buf = torch.zeros(5, dtype=torch.int32, device="cuda")
    assert J().jab_selftest_bounds_check(buf, 4) == 2  # JAB_ERR_UNSUPPORTED: nothing launched
    assert J().jab_get_device_status() == 0


def test_parity_cases_raise_no_check_in_the_checked_build():
    """Forward (teacher, loss), KL, Hutchinson, backward (with and without the KL term), weight
    gradient and the CTA-pair GEMMs on
    small cases, each test asserting its parity bar and device status 0, on libjab_checked.so."""
    r = _child([sys.executable, "-m", "pytest", "-x", "-q", "-m", "gpu", "-p", "no:cacheprovider",
                os.path.join("tests", "test_gpu_parity.py"), "-k",
                "teacher_output_parity or loss_forward_parity or backward_parity or backward_kl or "
                "weight_gradient_and_fisher or kl_forward or hutchinson or bit_identical"])
    assert r.returncode == 0, r.stdout[-3000:] + r.stderr[-3000:]
