"""Parity at the full sizes of the five workloads, in the launch configuration bench.py times.

The oracle cannot process a whole Mistral-sized batch, so it checks what it can compute one by
one: sequences are independent, so the GPU's per-(sequence, head) SSE of sampled sequences must
match the oracle run on those sequences alone; the scale gradient is checked on a sub-batch, and
the full-batch gradient by shard additivity (it is a size-weighted sum over sequence shards).
"""
import numpy as np
import pytest
import torch

from oracle import jab_oracle as O
from tests.harness import COS_MIN, L_TOL, J, cosine, np64, oracle_desc
from workloads import WORKLOADS, make_block_weights, make_x

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_34866_gb300 import build
    build.build()
    J().jab_get_device_status()
    yield


def _setup(name, block=0):
    wl = WORKLOADS[name]
    desc = J().desc_from_shape(wl.shape, wl.group_size)
    X = make_x(wl, device="cuda")
    W = make_block_weights(wl, block, device="cuda")
    return wl, desc, X, W


def _teacher(wl, desc, X, W, ws):
    A = torch.empty((wl.batch, wl.seq_len, wl.shape.n_q_heads * wl.shape.head_dim),
                    dtype=torch.float32, device="cuda")
    J().jab_reference_forward(desc, wl.batch, wl.seq_len, X, W, A, ws)
    return A


def _scales(desc, wl, W, bits):
    mode = 1 if wl.scale_init == "minmse" else 0
    s = torch.empty((wl.shape.d_out, wl.shape.d_model // wl.group_size), dtype=torch.float32,
                    device="cuda")
    J().jab_init_scales(desc, bits, mode, W, s)
    return s


def _check_sampled_sse(wl, X, W, scales, bits, parts, samples):
    od = oracle_desc(wl.shape, wl.group_size)
    w64 = np64(W)
    for b in samples:
        x64 = np64(X[b:b + 1])
        a_ref = O.block_forward(x64, w64, od)
        for i, (bb, s) in enumerate(zip(bits, scales)):
            r = O.jab_loss(x64, w64, s.cpu().numpy(), bb, od, a_ref=a_ref)
            got = parts[i, b].cpu().numpy()
            assert abs(got.sum() - r["sse"]) <= L_TOL * r["sse"], (bb, b, got.sum(), r["sse"])


def _forward_full(name, samples, block=0):
    wl, desc, X, W = _setup(name, block)
    ws = J().Workspace(desc, wl.batch, wl.seq_len, len(wl.bits), False)
    A = _teacher(wl, desc, X, W, ws)
    scales = [_scales(desc, wl, W, b) for b in wl.bits]
    loss = torch.empty(len(wl.bits), dtype=torch.float64, device="cuda")
    parts = torch.empty((len(wl.bits), wl.batch, wl.shape.n_q_heads), dtype=torch.float64,
                        device="cuda")
    J().jab_loss_forward(desc, wl.batch, wl.seq_len, X, W, A, list(wl.bits), scales, loss, ws,
                         sse_parts=parts)
    assert J().jab_get_device_status() == 0
    n = wl.batch * wl.seq_len * wl.shape.n_q_heads * wl.shape.head_dim
    np.testing.assert_allclose(loss.cpu().numpy(), parts.sum(dim=(1, 2)).cpu().numpy() / n,
                               rtol=1e-12)
    _check_sampled_sse(wl, X, W, scales, wl.bits, parts, samples)


def test_gpt2_sweep_forward_full_size():
    _forward_full("gpt2_sweep", samples=[0, 37])


def test_mistral_block_forward_full_size():
    _forward_full("mistral_block", samples=[5])


@pytest.mark.parametrize("block", [0, 31])
def test_mistral_scoring_forward_full_size(block):
    _forward_full("mistral_scoring", samples=[11], block=block)


def _backward(wl, desc, X, W, A, s, bits, B):
    ws = J().Workspace(desc, B, wl.seq_len, 1, True)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    g = torch.empty_like(s)
    J().jab_loss_backward_scales(desc, B, wl.seq_len, X[:B].contiguous(), W, A[:B].contiguous(),
                                 bits, s, 1.0, loss, g, ws)
    return loss.item(), g


@pytest.mark.parametrize("name,k", [("gpt2_smoke", 4), ("mistral_block", 1), ("mistral_ste_long", 1)])
def test_backward_full_size(name, k):
    wl, desc, X, W = _setup(name)
    bits = wl.bits[0]
    ws = J().Workspace(desc, wl.batch, wl.seq_len, 1, True)
    A = _teacher(wl, desc, X, W, ws)
    del ws
    s = _scales(desc, wl, W, bits)
    loss_full, g_full = _backward(wl, desc, X, W, A, s, bits, wl.batch)
    # sub-batch of k sequences against the oracle
    loss_k, g_k = _backward(wl, desc, X, W, A, s, bits, k)
    od = oracle_desc(wl.shape, wl.group_size)
    r = O.jab_loss_and_grad(np64(X[:k]), np64(W), s.cpu().numpy(), bits, od, kappa=1.0)
    assert abs(loss_k - r["loss"]) <= L_TOL * r["loss"], (loss_k, r["loss"])
    assert cosine(g_k.cpu().numpy(), r["grad_s"]) >= COS_MIN
    # shard additivity of the full batch: two halves, size-weighted
    if wl.batch >= 2:
        h = wl.batch // 2
        l1, g1 = _backward(wl, desc, X, W, A, s, bits, h)
        X2, A2 = X[h:].contiguous(), A[h:].contiguous()
        ws2 = J().Workspace(desc, wl.batch - h, wl.seq_len, 1, True)
        loss2 = torch.empty(1, dtype=torch.float64, device="cuda")
        g2 = torch.empty_like(s)
        J().jab_loss_backward_scales(desc, wl.batch - h, wl.seq_len, X2, W, A2, bits, s, 1.0, loss2,
                                     g2, ws2)
        f1, f2 = h / wl.batch, (wl.batch - h) / wl.batch
        np.testing.assert_allclose(loss_full, f1 * l1 + f2 * loss2.item(), rtol=1e-9)
        comb = (f1 * g1 + f2 * g2).cpu().numpy()
        assert cosine(g_full.cpu().numpy(), comb) >= 0.99999
    assert J().jab_get_device_status() == 0
