"""The C-ABI library loads and exports every entry point include/jab.h declares (no GPU needed),
and the host-side argument checks answer without touching a device."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "jab.h")


def _declared_symbols():
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(jab_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def libjab():
    from paper_2609_34866_gb300 import build
    build.build()
    return ctypes.CDLL(build.LIB_PATH)


def test_header_declares_the_boundary():
    syms = _declared_symbols()
    for name in ("jab_reference_forward", "jab_loss_forward", "jab_loss_backward_scales",
                 "jab_loss_backward_weights",
                 "jab_workspace_size", "jab_quantize", "jab_init_scales", "jab_get_device_status",
                 "jab_status_string"):
        assert name in syms


def test_library_exports_every_declared_symbol(libjab):
    missing = [s for s in _declared_symbols() if not hasattr(libjab, s)]
    assert not missing, missing


def test_host_side_checks_without_gpu(libjab):
    from paper_2609_34866_gb300 import binding as J
    J._LIB = None
    L = J.lib()
    good = J.BlockDesc(4096, 32, 8, 128, 128, 1, 10000.0, 0.0)
    n = J.jab_workspace_size(good, 2, 130, 5, True)
    assert n > 2 * 130 * 4096 * 2
    assert J.jab_workspace_size(good, 2, 130, 5, True) >= J.jab_workspace_size(good, 2, 130, 1, False)
    bad_dh = J.BlockDesc(4096, 32, 8, 96, 128, 1, 10000.0, 0.0)
    assert J.jab_workspace_size(bad_dh, 2, 130, 1, True) == 0
    bad_g = J.BlockDesc(4096, 32, 8, 128, 100, 1, 10000.0, 0.0)
    assert J.jab_workspace_size(bad_g, 2, 130, 1, True) == 0
    assert J.jab_workspace_size(good, 0, 130, 1, True) == 0
    # NULL pointers are rejected on the host before any CUDA call
    st = L.jab_loss_backward_scales(ctypes.byref(good), 2, 130, None, None, None, 3, None, 1.0,
                                    None, None, None, 0, None)
    assert st == 1
    # neither a gradient nor its norm requested
    st = L.jab_loss_backward_weights(ctypes.byref(good), 2, 130, None, None, None, 2, None, None,
                                     None, None, None, 0, None)
    assert st == 1
    st = L.jab_loss_backward_scales_prepared(ctypes.byref(good), 2, 130, None, None, None, 3, None,
                                             1.0, None, None, None, 0, None)
    assert st == 1
    assert L.jab_prepare_x(ctypes.byref(good), 2, 130, None, None, 0, None) == 1
    # the KL-term backward: no teacher projection / log-sum-exp, a negative or NaN lambda, an
    # unsupported block, each refused before any CUDA call
    fake = ctypes.c_void_p(1 << 20)  # never dereferenced: the checks fail first
    st = L.jab_loss_backward_scales_kl(ctypes.byref(good), 2, 130, fake, fake, fake, None, fake, 3,
                                       fake, 1.0, 0.1, fake, None, fake, fake, 1 << 40, None)
    assert st == 1
    st = L.jab_loss_backward_scales_kl(ctypes.byref(good), 2, 130, fake, fake, fake, fake, None, 3,
                                       fake, 1.0, 0.1, fake, None, fake, fake, 1 << 40, None)
    assert st == 1
    for lam in (-0.1, float("nan")):
        st = L.jab_loss_backward_scales_kl(ctypes.byref(good), 2, 130, fake, fake, fake, fake, fake,
                                           3, fake, 1.0, lam, fake, None, fake, fake, 1 << 40, None)
        assert st == 1
    st = L.jab_loss_backward_scales_kl(ctypes.byref(bad_dh), 2, 130, fake, fake, fake, fake, fake,
                                       3, fake, 1.0, 0.1, fake, None, fake, fake, 1 << 40, None)
    assert st == 2
    # the backward workspace holds the KL term's teacher log-sum-exp and partials too
    assert J.jab_workspace_size(good, 2, 130, 1, True) > J.jab_workspace_size(good, 2, 130, 1, False)
    assert L.jab_flip_rate(None, None, 16, None, None) == 1
    assert L.jab_selftest_bounds_check(None, 4, None) == 1
    assert L.jab_set_deterministic(2) == 1 and L.jab_set_deterministic(0) == 0
    st = L.jab_quantize(ctypes.byref(bad_dh), 3, None, None, None, None, None)
    assert st == 2
    assert L.jab_status_string(4).decode() == "non-finite or non-positive value"
