"""The seeded synthetic inputs (workloads/): determinism, the prefix property the sampled-sequence
parity tests rely on, and the documented value distributions, checked against closed forms."""
import math
from dataclasses import replace

import numpy as np
import pytest
import torch

from workloads import WORKLOADS, make_block_weights, make_x


def test_inputs_are_deterministic_and_seed_dependent():
    wl = WORKLOADS["gpt2_smoke"]
    a, b = make_x(wl), make_x(wl)
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    assert not torch.equal(make_x(wl, seed=1), a)
    assert torch.equal(make_block_weights(wl).view(torch.int16), make_block_weights(wl).view(torch.int16))


def test_first_sequences_do_not_depend_on_the_batch_size():
    wl = WORKLOADS["mistral_ste_long"]
    small = make_x(wl, batch=1, seq_len=16)
    large = make_x(wl, batch=3, seq_len=16)
    assert torch.equal(small[0].view(torch.int16), large[0].view(torch.int16))


@pytest.mark.parametrize("name", ["mistral_block", "mistral_ste_long"])
def test_student_t_activations_have_the_stated_scale_and_outliers(name):
    """Median |x| of unit-variance Student-t(df) is t_df^{-1}(0.75) / sqrt(df / (df - 2)); the
    outlier channels (ceil(p d) of them) carry that median times the stated factor."""
    stats = pytest.importorskip("scipy.stats")
    wl = WORKLOADS[name]
    x = make_x(wl, batch=1, seq_len=512)[0].float().numpy()
    d = wl.shape.d_model
    med = np.median(np.abs(x), axis=0)                            # per channel
    expect = stats.t.ppf(0.75, wl.x_df) / math.sqrt(wl.x_df / (wl.x_df - 2.0))
    n_out = int(math.ceil(wl.outlier_frac * d)) if wl.outlier_frac > 0 else 0
    heavy = med > 0.5 * wl.outlier_factor * expect if n_out else np.zeros(d, bool)
    assert int(heavy.sum()) == n_out
    np.testing.assert_allclose(np.median(np.abs(x[:, ~heavy])), expect, rtol=0.02)
    if n_out:
        np.testing.assert_allclose(np.median(np.abs(x[:, heavy])) / expect, wl.outlier_factor,
                                   rtol=0.05)


def test_normal_activations_and_weights():
    wl = replace(WORKLOADS["gpt2_sweep"], outlier_frac=0.0)
    x = make_x(wl, batch=1, seq_len=512).float().numpy()
    assert abs(x.mean()) < 0.01 and abs(x.std() - 1.0) < 0.01
    w = make_block_weights(WORKLOADS["mistral_block"]).float().numpy()
    assert w.shape == (WORKLOADS["mistral_block"].shape.d_out, 4096)
    np.testing.assert_allclose(w.std(), WORKLOADS["mistral_block"].w_std, rtol=0.01)
    assert abs(w.mean()) < 1e-4
