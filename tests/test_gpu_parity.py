"""GPU parity: the C-ABI path against the float64 oracle on the same seeded inputs.

Bars: integer codes bit-exact; attention output within 1e-2 of its RMS; L_JAB relative error
<= 1e-2; scale-gradient cosine >= 0.999 (fp16 tensor-core operands, fp32 accumulation).
"""
import numpy as np
import pytest
import torch

from oracle import jab_oracle as O
from tests.harness import A_TOL, COS_MIN, L_TOL, SMALL_CASES, Case, J, cosine, np64

pytestmark = pytest.mark.gpu

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_34866_gb300 import build
    build.build()
    J().jab_get_device_status()
    yield
    assert J().jab_get_device_status() == 0


_cases = {}


def case(name) -> Case:
    if name not in _cases:
        wl, B, T, G = SMALL_CASES[name]
        _cases[name] = Case(wl, B, T, G)
    return _cases[name]


# ------------------------------------------------------------------ quantiser: bit-exact
@pytest.mark.parametrize("name", ["gpt2_T200", "mistral_G64_T70"])
@pytest.mark.parametrize("bits", [2, 3, 4, 5, 8])
def test_quantize_codes_bit_exact(name, bits):
    c = case(name)
    s = c.gpu_scales(bits) * 0.8           # some codes clamp
    codes = torch.empty(c.W.shape, dtype=torch.int8, device="cuda")
    w_hat = torch.empty(c.W.shape, dtype=torch.float32, device="cuda")
    J().jab_quantize(c.desc, bits, c.W, s, codes=codes, w_hat=w_hat)
    oc, ow, _ = O.quantize(c.w64, s.cpu().numpy(), bits, c.G)
    np.testing.assert_array_equal(codes.cpu().numpy(), oc)
    np.testing.assert_array_equal(w_hat.cpu().numpy(), ow.astype(np.float32))
    assert J().jab_get_device_status() == 0


@pytest.mark.parametrize("bits", [2, 3, 8])
def test_init_scales(bits):
    c = case("mistral_G64_T70")
    s0 = c.gpu_scales(bits, mode=0).cpu().numpy()
    np.testing.assert_array_equal(s0, O.init_scales_absmax(c.w64, bits, c.G))
    s1 = c.gpu_scales(bits, mode=1).cpu().numpy()
    so = O.init_scales_minmse(c.w64, bits, c.G)

    def crit(s):
        _, wh, _ = O.quantize(c.w64, s, bits, c.G)
        return ((wh - c.w64) ** 2).reshape(c.D, -1, c.G).sum(axis=2)

    cg, co = crit(s1), crit(so)
    # the choice may differ only where two candidates tie to rounding in the criterion
    assert np.all(cg <= co * (1 + 1e-6) + 1e-30)
    assert (s1 == so).mean() > 0.999


# ------------------------------------------------------------------ teacher output
@pytest.mark.parametrize("name", list(SMALL_CASES))
def test_teacher_output_parity(name):
    c = case(name)
    A, lse, sq = c.gpu_teacher()
    a_o, parts = O.block_forward(c.x64, c.w64, c.odesc, return_parts=True)
    A = np64(A)
    rms = np.sqrt((a_o ** 2).mean())
    err_rms = np.sqrt(((A - a_o) ** 2).mean())
    assert err_rms <= A_TOL * rms, (err_rms, rms)                    # the bar: error RMS / RMS
    assert np.abs(A - a_o).max() <= A_TOL * np.abs(a_o).max()       # and element-wise vs. max
    np.testing.assert_allclose(np64(lse), parts["lse"], rtol=1e-3, atol=1e-2)  # fp16 Q, K scores
    np.testing.assert_allclose(sq.item(), (a_o ** 2).sum(), rtol=2e-3)


# ------------------------------------------------------------------ forward loss over candidates
@pytest.mark.parametrize("name", ["gpt2_T200", "mistral_T130", "gqa2_T257", "dh64_gqa4_T65",
                                  "dh64_gqa4_B64_T256", "gpt2_T1"])
def test_loss_forward_parity(name):
    c = case(name)
    ws = c.workspace(n_cand=5)
    A, _, _ = c.gpu_teacher(ws)
    bits = [2, 3, 4, 5, 8]
    scales = [c.gpu_scales(b) for b in bits]
    loss = torch.empty(len(bits), dtype=torch.float64, device="cuda")
    parts = torch.empty((len(bits), c.B, c.Hq), dtype=torch.float64, device="cuda")
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, c.W, A, bits, scales, loss, ws, sse_parts=parts)
    a_ref = c.oracle_teacher()
    for i, b in enumerate(bits):
        r = O.jab_loss(c.x64, c.w64, scales[i].cpu().numpy(), b, c.odesc, a_ref=a_ref)
        assert abs(loss[i].item() - r["loss"]) <= L_TOL * r["loss"], (b, loss[i].item(), r["loss"])
        np.testing.assert_allclose(parts[i].cpu().numpy(), r["sse_parts"], rtol=5e-2)
        np.testing.assert_allclose(parts[i].sum().item(), r["sse"], rtol=L_TOL)
    assert J().jab_get_device_status() == 0


# ------------------------------------------------------------------ STE / LSQ backward
@pytest.mark.parametrize("name,bits", [("gpt2_T200", 3), ("mistral_T130", 3),
                                       ("mistral_G64_T70", 2), ("gqa2_T257", 3),
                                       ("dh64_gqa4_T65", 4), ("dh64_gqa4_B64_T256", 3),
                                       ("gpt2_T1", 3)])
def test_backward_parity(name, bits):
    c = case(name)
    ws = c.workspace()
    A, _, _ = c.gpu_teacher(ws)
    s = c.gpu_scales(bits)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    grad = torch.empty_like(s)
    J().jab_loss_backward_scales(c.desc, c.B, c.T, c.X, c.W, A, bits, s, 1.0, loss, grad, ws)
    r = O.jab_loss_and_grad(c.x64, c.w64, s.cpu().numpy(), bits, c.odesc, a_ref=c.oracle_teacher(),
                            kappa=1.0)
    assert abs(loss.item() - r["loss"]) <= L_TOL * r["loss"]
    g = grad.cpu().numpy()
    if c.T == 1:   # softmax over one key: Q and K scale gradients vanish (here to fp32 rounding:
        # dP - rowsum(dO * O) cancels only up to the summation order of the two dot products)
        nqk = (c.Hq + c.shape.n_kv_heads) * c.dh
        assert np.abs(g[:nqk]).max() <= 1e-4 * np.abs(g[nqk:]).max()
    assert cosine(g, r["grad_s"]) >= COS_MIN, cosine(g, r["grad_s"])
    # kappa <= 0 selects (G qmax)^(-1/2): a pure multiplier
    grad2 = torch.empty_like(s)
    J().jab_loss_backward_scales(c.desc, c.B, c.T, c.X, c.W, A, bits, s, 0.0, loss, grad2, ws)
    k = 1.0 / np.sqrt(c.G * ((1 << (bits - 1)) - 1))
    # (fp32 atomics: the summation order differs between calls)
    np.testing.assert_allclose(grad2.cpu().numpy(), g * k, rtol=1e-4, atol=1e-5 * np.abs(g * k).max())
    assert J().jab_get_device_status() == 0


# ------------------------------------------------------------------ STE weight gradient, Fisher score
@pytest.mark.parametrize("name,bits", [("gpt2_T200", 2), ("mistral_T130", 2), ("gqa2_T257", 3),
                                       ("dh64_gqa4_B64_T256", 2)])
def test_weight_gradient_and_fisher_coupling_score(name, bits):
    """dL/dw_hat (App. B, STE) against the oracle's finite-difference-pinned gradient, and its squared
    norm: with bits = 2 and absmax (round-to-nearest) scales, the Fisher-coupling score (App. B)."""
    c = case(name)
    ws = c.workspace()
    A, _, _ = c.gpu_teacher(ws)
    s = c.gpu_scales(bits, mode=0)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    gw = torch.empty(c.W.shape, dtype=torch.float32, device="cuda")
    sq = torch.empty(1, dtype=torch.float64, device="cuda")
    J().jab_loss_backward_weights(c.desc, c.B, c.T, c.X, c.W, A, bits, s, loss, grad_w=gw,
                                  grad_sqnorm=sq, ws=ws)
    r = O.jab_loss_and_grad(c.x64, c.w64, s.cpu().numpy(), bits, c.odesc, a_ref=c.oracle_teacher(),
                            kappa=1.0)
    assert abs(loss.item() - r["loss"]) <= L_TOL * r["loss"]
    g, go = np64(gw), r["grad_w_hat"]
    assert cosine(g, go) >= COS_MIN, cosine(g, go)
    # the norm matches the stored gradient's own (fp64 sum of the same fp32 values, other order) ...
    np.testing.assert_allclose(sq.item(), (g ** 2).sum(), rtol=1e-5)
    # ... and the oracle's within the gradient's error (|g|^2 = |go|^2 (1 + O(err^2)))
    np.testing.assert_allclose(sq.item(), (go ** 2).sum(), rtol=2e-2)
    # the score alone, without storing the gradient
    sq2 = torch.empty(1, dtype=torch.float64, device="cuda")
    J().jab_loss_backward_weights(c.desc, c.B, c.T, c.X, c.W, A, bits, s, loss, grad_sqnorm=sq2, ws=ws)
    np.testing.assert_allclose(sq2.item(), sq.item(), rtol=1e-6)
    assert J().jab_get_device_status() == 0


def test_weight_gradient_vanishes_on_grid():
    """Weights on the grid: student = teacher, so L = 0, dL/dw_hat = 0 and the score is 0 exactly."""
    c = case("mistral_T130")
    rng = np.random.default_rng(1)
    q = rng.integers(-1, 2, size=c.W.shape)
    W = torch.tensor(q * 2.0 ** -6, dtype=torch.bfloat16, device="cuda")
    s = torch.full((c.D, c.shape.d_model // c.G), 2.0 ** -6, dtype=torch.float32, device="cuda")
    ws = c.workspace()
    A = torch.empty((c.B, c.T, c.Hq * c.dh), dtype=torch.float32, device="cuda")
    J().jab_reference_forward(c.desc, c.B, c.T, c.X, W, A, ws)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    gw = torch.full(W.shape, 7.0, dtype=torch.float32, device="cuda")
    sq = torch.full((1,), 7.0, dtype=torch.float64, device="cuda")
    J().jab_loss_backward_weights(c.desc, c.B, c.T, c.X, W, A, 2, s, loss, grad_w=gw, grad_sqnorm=sq,
                                  ws=ws)
    assert loss.item() == 0.0 and sq.item() == 0.0 and not gw.any()


# ------------------------------------------------------------------ exact special cases
def test_loss_exactly_zero_on_grid():
    """Weights on the grid: the student is the teacher bit for bit, so L = 0 and grad = 0."""
    c = case("mistral_T130")
    rng = np.random.default_rng(0)
    q = rng.integers(-3, 4, size=c.W.shape)
    W = torch.tensor(q * 2.0 ** -7, dtype=torch.bfloat16, device="cuda")
    s = torch.full((c.D, c.shape.d_model // c.G), 2.0 ** -7, dtype=torch.float32, device="cuda")
    ws = c.workspace()
    A = torch.empty((c.B, c.T, c.Hq * c.dh), dtype=torch.float32, device="cuda")
    J().jab_reference_forward(c.desc, c.B, c.T, c.X, W, A, ws)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, W, A, [3], [s], loss, ws)
    assert loss.item() == 0.0
    grad = torch.empty_like(s)
    J().jab_loss_backward_scales(c.desc, c.B, c.T, c.X, W, A, 3, s, 1.0, loss, grad, ws)
    assert loss.item() == 0.0 and not grad.any()


def test_repeated_calls_are_bit_identical():
    c = case("gpt2_T200")
    ws = c.workspace(n_cand=2)
    A, _, _ = c.gpu_teacher(ws)
    s = [c.gpu_scales(2), c.gpu_scales(4)]
    l1 = torch.empty(2, dtype=torch.float64, device="cuda")
    l2 = torch.empty(2, dtype=torch.float64, device="cuda")
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, c.W, A, [2, 4], s, l1, ws)
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, c.W, A, [2, 4], s, l2, ws)
    assert torch.equal(l1, l2)


# ------------------------------------------------------------------ error paths (no GPU fault)
def test_error_paths():
    c = case("gpt2_T200")
    ws = c.workspace()
    A, _, _ = c.gpu_teacher(ws)
    s = c.gpu_scales(3)
    loss = torch.empty(1, dtype=torch.float64, device="cuda")
    grad = torch.empty_like(s)
    small = J().Workspace(c.desc, 1, 1, 1, False)
    with pytest.raises(J().JabError) as e:
        J().jab_loss_backward_scales(c.desc, c.B, c.T, c.X, c.W, A, 3, s, 1.0, loss, grad, small)
    assert e.value.status == 1
    with pytest.raises(J().JabError) as e:
        J().jab_loss_backward_scales(c.desc, c.B, c.T, c.X, c.W, A, 9, s, 1.0, loss, grad, ws)
    assert e.value.status == 1
    bad = s.clone()
    bad[3, 1] = 0.0                                   # a non-positive scale is reported, not used
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, c.W, A, [3], [bad], loss, ws)
    assert J().jab_get_device_status() == 4
    bad[3, 1] = float("nan")
    J().jab_loss_forward(c.desc, c.B, c.T, c.X, c.W, A, [3], [bad], loss, ws)
    assert J().jab_get_device_status() == 4
    X = c.X.clone()
    X[0, 5, 7] = 1.0e5                                # outside the fp16 range of the fp16 operands
    J().jab_loss_forward(c.desc, c.B, c.T, X, c.W, A, [3], [s], loss, ws)
    assert J().jab_get_device_status() == 5
    assert J().jab_get_device_status() == 0


def test_bounded_wait_times_out_and_context_survives():
    """A pipelined kernel's wait on a barrier that never flips gives up after its limit, reports
    JAB_ERR_TIMEOUT through the status word, and later calls still work (no fault, no hang)."""
    J().jab_get_device_status()
    J().jab_selftest_wait_timeout()
    assert J().jab_get_device_status() == 6
    c = case("gpt2_T1")
    A, _, _ = c.gpu_teacher()
    assert J().jab_get_device_status() == 0
    np.testing.assert_allclose(np64(A), c.oracle_teacher(), rtol=0, atol=1e-2 * np.abs(c.oracle_teacher()).max())
