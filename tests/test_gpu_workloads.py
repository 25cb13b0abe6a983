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
from tests.harness import A_TOL, COS_MIN, HEAVY_MAX_ERR, L_TOL, J, cosine, np64, oracle_desc
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


def _check_sampled_sse(wl, X, W, A, scales, bits, parts, samples):
    od = oracle_desc(wl.shape, wl.group_size)
    w64 = np64(W)
    for b in samples:
        x64 = np64(X[b:b + 1])
        a_ref = O.block_forward(x64, w64, od)
        # the full-batch teacher output of this sequence, element by element
        err = np.abs(np64(A[b]) - a_ref[0])
        rms = np.sqrt((a_ref ** 2).mean())
        assert np.sqrt((err ** 2).mean()) <= A_TOL * rms, (b, np.sqrt((err ** 2).mean()) / rms)
        if wl.x_dist == "normal":
            assert err.max() <= A_TOL * rms, (b, err.max() / rms)
        else:
            # Heavy-tailed X: the scores of outlier rows are large, so the fp16 rounding of Q and K
            # shifts their softmax weights, and an output entry's error follows the spread of V over
            # its row rather than its own size (measured max|err| / RMS: 1.2e-2 on the 128 x 2048
            # block, 3.9e-2 on the scoring batch, 4.9e-2 on the long-context batch)
            assert err.max() <= HEAVY_MAX_ERR * rms, (b, err.max() / rms)
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
    _check_sampled_sse(wl, X, W, A, scales, wl.bits, parts, samples)


def test_gpt2_sweep_forward_full_size():
    _forward_full("gpt2_sweep", samples=[0, 37])


def test_mistral_block_forward_full_size():
    _forward_full("mistral_block", samples=[5])


def test_mistral_ste_long_forward_full_size():
    _forward_full("mistral_ste_long", samples=[3])


@pytest.mark.parametrize("block", [0, 31])
def test_mistral_scoring_forward_full_size(block):
    _forward_full("mistral_scoring", samples=[11], block=block)


def test_mistral_scoring_kl_full_size():
    """The KL term of Eq. 3 over all five candidates of the scoring workload at full size; one
    sampled sequence's rows against the oracle run on that sequence alone (rows are independent)."""
    from tests.harness import KL_ROW_ATOL, KL_ROW_TOL, KL_TOL
    wl, desc, X, W = _setup("mistral_scoring")
    ws = J().Workspace(desc, wl.batch, wl.seq_len, len(wl.bits), False)
    A = _teacher(wl, desc, X, W, ws)
    qkv_ref = torch.empty((wl.batch, wl.seq_len, wl.shape.d_out), dtype=torch.float16, device="cuda")
    J().jab_reference_projection(desc, wl.batch, wl.seq_len, X, W, qkv_ref, ws)
    scales = [_scales(desc, wl, W, b) for b in wl.bits]
    C = len(wl.bits)
    loss, mse, kl = (torch.empty(C, dtype=torch.float64, device="cuda") for _ in range(3))
    rows = torch.empty((C, wl.batch, wl.shape.n_q_heads, wl.seq_len), dtype=torch.float32,
                       device="cuda")
    J().jab_loss_forward_kl(desc, wl.batch, wl.seq_len, X, W, A, qkv_ref, list(wl.bits), scales, 0.1,
                            loss, ws, mse=mse, kl=kl, kl_rows=rows)
    assert J().jab_get_device_status() == 0
    np.testing.assert_allclose(kl.cpu().numpy(), rows.double().sum(dim=(1, 2, 3)).cpu().numpy() / wl.batch,
                               rtol=1e-5)
    od = oracle_desc(wl.shape, wl.group_size)
    b = 11
    for i, bits in enumerate(wl.bits):
        r = O.kl_attention_term(np64(X[b:b + 1]), np64(W), scales[i].cpu().numpy(), bits, od)
        ro, got = r["kl_rows"][0], np64(rows[i, b])
        assert abs(got.sum() - ro.sum()) <= KL_TOL[bits] * ro.sum(), (bits, got.sum(), ro.sum())
        if bits in KL_ROW_TOL:
            bound = KL_ROW_TOL[bits] * (ro + ro.mean()) + KL_ROW_ATOL
            assert (np.abs(got - ro) <= bound).all(), (bits, (np.abs(got - ro) / bound).max())


def test_mistral_scoring_hutchinson_full_sequence():
    """The Hutchinson quadratic form on one full-length sequence of the scoring workload's block
    (T = 2048, d_model 4096, GQA 32/8, RoPE), one probe, against the oracle on that sequence."""
    from tests.harness import JVP_TOL
    wl, desc, X, W = _setup("mistral_scoring")
    x1 = X[:1].contiguous()
    ws = J().Workspace(desc, 1, wl.seq_len, 2, False)
    A = torch.empty((1, wl.seq_len, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32,
                    device="cuda")
    lse = torch.empty((1, wl.shape.n_q_heads, wl.seq_len), dtype=torch.float32, device="cuda")
    J().jab_reference_forward(desc, 1, wl.seq_len, x1, W, A, ws, lse=lse)
    trace = torch.empty(1, dtype=torch.float64, device="cuda")
    J().jab_hutchinson_trace(desc, 1, wl.seq_len, x1, W, A, lse, 1, 77, trace, ws)
    assert J().jab_get_device_status() == 0
    v = O.rademacher_probe(77, 0, tuple(W.shape))
    want = O.gn_quadratic_form(np64(x1), np64(W), v, oracle_desc(wl.shape, wl.group_size))
    assert abs(trace.item() - want) <= JVP_TOL * want, (trace.item(), want)


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


def test_backward_kl_full_size():
    """The STE backward of both terms of Eq. 3 (lambda_KL = 0.1) on the Mistral-7B-shaped block at
    its full size (the launch bench.py times): a one-sequence sub-batch against the oracle's joint
    gradient, and the full batch against its two halves (the batchmean KL is the mean of the
    halves', the loss and the gradient their size-weighted sums)."""
    wl, desc, X, W = _setup("mistral_block")
    bits, lam = wl.bits[0], float(np.float32(0.1))
    s = _scales(desc, wl, W, bits)
    T = wl.seq_len

    def run(Xb, nb):
        ws = J().Workspace(desc, nb, T, 1, True)
        A = torch.empty((nb, T, wl.shape.n_q_heads * wl.shape.head_dim), dtype=torch.float32,
                        device="cuda")
        lse = torch.empty((nb, wl.shape.n_q_heads, T), dtype=torch.float32, device="cuda")
        J().jab_reference_forward(desc, nb, T, Xb, W, A, ws, lse=lse)
        qkv_ref = torch.empty((nb, T, wl.shape.d_out), dtype=torch.float16, device="cuda")
        J().jab_reference_projection(desc, nb, T, Xb, W, qkv_ref, ws)
        loss, kl = (torch.empty(1, dtype=torch.float64, device="cuda") for _ in range(2))
        g = torch.empty_like(s)
        J().jab_loss_backward_scales_kl(desc, nb, T, Xb, W, A, qkv_ref, lse, bits, s, 1.0, lam,
                                        loss, g, ws, kl=kl)
        assert J().jab_get_device_status() == 0
        return loss.item(), kl.item(), g

    l_full, kl_full, g_full = run(X, wl.batch)
    l1, kl1, g1 = run(X[:1].contiguous(), 1)
    r = O.jab_loss_joint_and_grad(np64(X[:1]), np64(W), s.cpu().numpy(), bits,
                                  oracle_desc(wl.shape, wl.group_size), lam_kl=lam, kappa=1.0)
    assert abs(kl1 - r["kl"]) <= L_TOL * r["kl"], (kl1, r["kl"])
    assert abs(l1 - r["loss"]) <= L_TOL * r["loss"], (l1, r["loss"])
    assert cosine(g1.cpu().numpy(), r["grad_s"]) >= COS_MIN
    h = wl.batch // 2
    la, kla, ga = run(X[:h].contiguous(), h)
    lb, klb, gb = run(X[h:].contiguous(), wl.batch - h)
    np.testing.assert_allclose(kl_full, 0.5 * (kla + klb), rtol=1e-9)
    np.testing.assert_allclose(l_full, 0.5 * (la + lb), rtol=1e-9)
    comb = (0.5 * (ga + gb)).cpu().numpy()
    assert cosine(g_full.cpu().numpy(), comb) >= 0.99999


def test_weight_gradient_split_k_full_shape():
    """The STE weight gradient (App. B) on the Mistral-7B-shaped block at 8 and 4 sequences, where
    the weight-gradient GEMM splits the token range (2-3 parts, partial tiles added with atomics):
    the gradient is additive over sequences (halves recombined by their size), and the norm-only
    call (through the workspace scratch) matches the stored gradient's norm."""
    wl, desc, X, W = _setup("mistral_block")
    B = 8
    X = X[:B].contiguous()
    bits = wl.bits[0]
    s = _scales(desc, wl, W, bits)

    def grad(Xb, nb):
        ws = J().Workspace(desc, nb, wl.seq_len, 1, True)
        A = torch.empty((nb, wl.seq_len, wl.shape.n_q_heads * wl.shape.head_dim),
                        dtype=torch.float32, device="cuda")
        J().jab_reference_forward(desc, nb, wl.seq_len, Xb, W, A, ws)
        loss = torch.empty(1, dtype=torch.float64, device="cuda")
        gw = torch.empty(W.shape, dtype=torch.float32, device="cuda")
        sq = torch.empty(1, dtype=torch.float64, device="cuda")
        J().jab_loss_backward_weights(desc, nb, wl.seq_len, Xb, W, A, bits, s, loss, grad_w=gw,
                                      grad_sqnorm=sq, ws=ws)
        sq2 = torch.empty(1, dtype=torch.float64, device="cuda")
        J().jab_loss_backward_weights(desc, nb, wl.seq_len, Xb, W, A, bits, s, loss, grad_sqnorm=sq2,
                                      ws=ws)
        g = gw.double()
        np.testing.assert_allclose(sq.item(), (g * g).sum().item(), rtol=1e-5)
        np.testing.assert_allclose(sq2.item(), sq.item(), rtol=1e-5)
        return g

    g_full = grad(X, B)
    h = B // 2
    g1 = grad(X[:h].contiguous(), h)
    g2 = grad(X[h:].contiguous(), B - h)
    comb = 0.5 * (g1 + g2)
    cos = (g_full * comb).sum() / (g_full.norm() * comb.norm())
    assert cos.item() >= 0.99999, cos.item()
    np.testing.assert_allclose(g_full.norm().item(), comb.norm().item(), rtol=1e-4)
    assert J().jab_get_device_status() == 0
