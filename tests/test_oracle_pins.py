"""Pins of the float64 oracle against what the paper and the mathematics fix (CPU only).

Each test names the passage it follows. None of them re-types the oracle's own formula:
they use hand-worked values, closed forms, invariances, brute force and finite differences.
"""
import json
import os

import numpy as np
import pytest

from oracle import jab_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _desc(d, Hq, Hkv, dh, G, rope=False, theta=10000.0):
    return dict(d_model=d, n_q_heads=Hq, n_kv_heads=Hkv, head_dim=dh, group_size=G,
                use_rope=rope, rope_theta=theta, softmax_scale=0.0)


def _bf16(a):
    """Round float64 values to bf16 (round-to-nearest-even), returned as float64."""
    a32 = np.asarray(a, dtype=np.float32)
    u = a32.view(np.uint32).astype(np.uint64)
    u = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def _tiny(seed=0, B=2, T=6, d=8, Hq=2, Hkv=1, dh=4, G=4, rope=False, w_std=0.3):
    rng = np.random.default_rng(seed)
    desc = _desc(d, Hq, Hkv, dh, G, rope)
    D = (Hq + 2 * Hkv) * dh
    x = _bf16(rng.standard_normal((B, T, d)))
    w = _bf16(rng.standard_normal((D, d)) * w_std)
    return desc, x, w


# ------------------------------------------------------------------ quantizer (Eq. 2, Eq. 13)

def test_quantizer_golden_worked_examples():
    with open(os.path.join(GOLDEN, "quantizer_worked.json")) as f:
        fx = json.load(f)
    for case in fx["cases"]:
        w = np.array([case["w"]])
        n = w.shape[1]
        s = np.array([[case["scale"]]], dtype=np.float32)
        codes, w_hat, v = O.quantize(w, s, case["bits"], n)
        assert codes[0].tolist() == case["codes"]
        np.testing.assert_array_equal(w_hat[0], case["w_hat"])
        np.testing.assert_array_equal(O.lsq_factor(v, case["bits"])[0], case["lsq"])


def _fp32_round_exact(x):
    """Correctly rounded binary32 value of a positive rational x (normal range), ties to even,
    by exact integer arithmetic (independent of numpy's float32 division)."""
    from fractions import Fraction
    x = Fraction(x)
    e = 0
    while x >= 2:
        x /= 2
        e += 1
    while x < 1:
        x *= 2
        e -= 1
    m = x * 2 ** 23
    fl, rem = divmod(m.numerator, m.denominator)
    rem = Fraction(rem, m.denominator)
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    return Fraction(fl, 2 ** 23) * Fraction(2) ** e


def test_quantizer_fp32_quotient_lands_on_half_integers():
    """Reading R1 of Eq. 2: the code is taken from the fp32 quotient. The fixture's scales are not
    powers of two and the exact quotients sit just off a half-integer that their fp32 rounding hits,
    so a float64 quotient (or any other rounding of w/s) gives a different code."""
    from fractions import Fraction
    with open(os.path.join(GOLDEN, "quantizer_worked.json")) as f:
        fx = json.load(f)["fp32_quotient_cases"]
    w = np.array([fx["w"]])
    s = np.array([[float.fromhex(h) for h in fx["scale_hex"]]], dtype=np.float32)
    for i, (num, den) in enumerate(fx["exact_quotient"]):       # the fixture's own arithmetic
        exact = Fraction(fx["w"][i]) / Fraction(float(s[0, i]))
        assert exact == Fraction(num, den)
        assert exact.denominator != 2 and _fp32_round_exact(exact) == Fraction(fx["v"][i])
        assert round(float(exact)) != fx["codes"][i]               # float64 quotient: other code
    codes, w_hat, v = O.quantize(w, s, fx["bits"], 1)
    assert codes[0].tolist() == fx["codes"]
    np.testing.assert_array_equal(v[0], fx["v"])
    np.testing.assert_array_equal(w_hat[0], [float.fromhex(h) for h in fx["w_hat_hex"]])
    np.testing.assert_array_equal(O.lsq_factor(v, fx["bits"])[0], fx["lsq"])


def test_flip_count_hand_worked():
    """Eq. 15 on six weights, b = 3, worked by hand. Before: s = 1/2, after: s = 3/8 (fp32-exact).
    w              = 0.3,   -0.55,  1.0, 0.1, 2.0, -1.6
    w / (1/2)      = 0.6,   -1.1,   2.0, 0.2, 4.0, -3.2   -> codes 1, -1, 2, 0, 3, -3
    w / (3/8)      = 0.8,   -1.466, 2.666, 0.266, 5.33, -4.266 -> codes 1, -1, 3, 0, 3, -3
    One grid position changes (1.0: 2 -> 3); 2.0 and -1.6 clamp to +-qmax on both sides."""
    w = np.array([[0.3, -0.55, 1.0, 0.1, 2.0, -1.6]])
    ca, _, _ = O.quantize(w, np.array([[0.5]], dtype=np.float32), 3, 6)
    cb, _, _ = O.quantize(w, np.array([[0.375]], dtype=np.float32), 3, 6)
    assert ca.tolist() == [[1, -1, 2, 0, 3, -3]] and cb.tolist() == [[1, -1, 3, 0, 3, -3]]
    assert O.flip_count(ca, cb) == 1 and O.flip_count(ca, ca) == 0


@pytest.mark.parametrize("bits", [2, 3, 4, 5, 8])
def test_quantizer_brute_force_nearest_grid_point(bits):
    """Eq. 2 equals the nearest point of {-qmax..qmax} to the fp32 quotient, ties to even."""
    rng = np.random.default_rng(bits)
    G = 16
    w = _bf16(rng.standard_normal((6, 64)) * 0.02)
    s = O.init_scales_absmax(w, bits, G) * np.float32(0.7)   # push some codes past the clamp
    codes, w_hat, v = O.quantize(w, s, bits, G)
    qm = (1 << (bits - 1)) - 1
    grid = np.arange(-qm, qm + 1)
    for idx in np.ndindex(w.shape):
        dist = np.abs(v[idx] - grid)
        best = np.flatnonzero(dist == dist.min())
        pick = best[0] if len(best) == 1 else [b for b in best if grid[b] % 2 == 0][0]
        assert codes[idx] == grid[pick], (idx, v[idx])
    assert codes.min() >= -qm and codes.max() <= qm
    assert (codes == qm).any() or (codes == -qm).any()


def test_quantizer_error_bound_idempotence_and_grid():
    rng = np.random.default_rng(1)
    G, bits = 8, 3
    w = _bf16(rng.standard_normal((4, 32)) * 0.05)
    s = O.init_scales_absmax(w, bits, G)
    codes, w_hat, v = O.quantize(w, s, bits, G)
    s_full = np.repeat(s.astype(np.float64), G, axis=1)
    inside = np.abs(v) <= (1 << (bits - 1)) - 1
    assert np.all(np.abs(w_hat - w)[inside] <= s_full[inside] / 2 * (1 + 1e-6))
    codes2, w_hat2, _ = O.quantize(w_hat, s, bits, G)          # Q(Q(w)) = Q(w)
    np.testing.assert_array_equal(codes2, codes)
    np.testing.assert_array_equal(w_hat2, w_hat)
    # weights built on the grid (powers-of-two scales, exact in bf16) reproduce their codes
    q = rng.integers(-3, 4, size=(4, 32))
    s_grid = np.full((4, 4), 2.0 ** -6, dtype=np.float32)
    w_grid = q * 2.0 ** -6
    c3, wh3, _ = O.quantize(w_grid, s_grid, bits, G)
    np.testing.assert_array_equal(c3, q)
    np.testing.assert_array_equal(wh3, w_grid)


def test_absmax_scale_init_maps_group_max_to_qmax():
    rng = np.random.default_rng(2)
    w = _bf16(rng.standard_normal((3, 16)) * 0.02)
    w[1, 8:] = 0.0                                   # all-zero group
    for bits in (2, 3, 8):
        s = O.init_scales_absmax(w, bits, 8)
        codes, _, _ = O.quantize(w, s, bits, 8)
        qm = (1 << (bits - 1)) - 1
        for o in range(3):
            for g in range(2):
                grp = np.abs(w[o, g * 8:(g + 1) * 8])
                if grp.max() == 0:
                    assert s[o, g] == 1.0 and not codes[o, g * 8:(g + 1) * 8].any()
                else:
                    assert np.abs(codes[o, g * 8:(g + 1) * 8]).max() == qm


def test_minmse_scale_search_brute_force():
    """Warm-start scales: the chosen scale attains the minimum over all candidates."""
    rng = np.random.default_rng(3)
    bits, G = 2, 8
    w = _bf16(rng.standard_normal((3, 16)) * 0.02)
    s = O.init_scales_minmse(w, bits, G)
    s0 = O.init_scales_absmax(w, bits, G).astype(np.float64)
    for o in range(3):
        for g in range(2):
            grp = w[o, g * G:(g + 1) * G]
            errs = []
            for k in range(80):
                sk = np.float32(s0[o, g] * (100 - k) / 100.0)
                c, wh, _ = O.quantize(grp[None], np.array([[sk]]), bits, G)
                errs.append(((wh[0] - grp) ** 2).sum())
            k_best = int(np.argmin(errs))
            assert s[o, g] == np.float32(s0[o, g] * (100 - k_best) / 100.0)
            assert errs[k_best] <= errs[0]


# ------------------------------------------------------------------ attention (Section 2.1)

def test_attention_golden_worked_example():
    with open(os.path.join(GOLDEN, "attention_worked.json")) as f:
        fx = json.load(f)
    desc = _desc(3, 1, 1, 1, 3)
    a = O.block_forward(np.array([fx["x"]]), np.array(fx["w"]), desc)
    np.testing.assert_allclose(a[0, :, 0], fx["a"], rtol=0, atol=1e-14)
    for case in fx["rope"]["cases"]:
        dh = case["head_dim"]
        cos, sin = O.rope_tables(case["t"] + 1, dh, 10000.0)
        x = np.zeros((1, case["t"] + 1, 1, dh))
        x[0, case["t"], 0] = case["x"]
        out = O.apply_rope(x, cos, sin)[0, case["t"], 0]
        np.testing.assert_allclose(out, case["out"], atol=1e-14)


def test_softmax_rows_and_causal_support():
    desc, x, w = _tiny(rope=True)
    a, parts = O.block_forward(x, w, desc, return_parts=True)
    P = parts["P"]
    np.testing.assert_allclose(P.sum(axis=-1), 1.0, atol=1e-13)
    assert (P >= 0).all()
    T = x.shape[1]
    assert np.all(P[..., np.triu_indices(T, 1)[0], np.triu_indices(T, 1)[1]] == 0)


def test_zero_query_weights_give_causal_running_mean():
    """W_Q = 0: every score is 0, so token t averages V over positions 0..t (GQA map h -> h//r)."""
    desc, x, w = _tiny(Hq=4, Hkv=2, dh=4, d=8, rope=True)
    w = w.copy()
    w[:16] = 0.0                                       # all query rows
    a = O.block_forward(x, w, desc)
    B, T, _ = x.shape
    v = (x @ w[24:32].T).reshape(B, T, 2, 4)           # V rows follow 16 Q rows and 8 K rows
    counts = np.arange(1, T + 1)[None, :, None, None]
    mean = np.cumsum(v, axis=1) / counts
    expect = np.concatenate([mean[:, :, h // 2] for h in range(4)], axis=-1)
    np.testing.assert_allclose(a, expect, atol=1e-13)


def test_causal_invariance_to_future_tokens():
    desc, x, w = _tiny(T=8, rope=True)
    s = O.init_scales_absmax(w, 3, desc["group_size"])
    r1 = O.jab_loss(x, w, s, 3, desc)
    x2 = x.copy()
    x2[:, 5:] = _bf16(np.random.default_rng(9).standard_normal(x2[:, 5:].shape))
    r2 = O.jab_loss(x2, w, s, 3, desc)
    np.testing.assert_array_equal(r1["a_ref"][:, :5], r2["a_ref"][:, :5])
    np.testing.assert_array_equal(r1["a_hat"][:, :5], r2["a_hat"][:, :5])
    assert not np.allclose(r1["a_ref"][:, 5:], r2["a_ref"][:, 5:])


def test_query_key_scaling_invariance_with_rope():
    """L_JAB depends on (W_Q, W_K) only through the scores; W_Q*c, W_K/c leaves A unchanged."""
    desc, x, w = _tiny(rope=True)
    a = O.block_forward(x, w, desc)
    w2 = w.copy()
    w2[:8] *= 4.0          # Q rows (Hq*dh = 8)
    w2[8:12] /= 4.0        # K rows
    np.testing.assert_allclose(O.block_forward(x, w2, desc), a, atol=1e-13)


def test_per_head_linear_invariance_without_rope():
    """Section 2.3 / App. B: W_Q -> W_Q R, W_K -> W_K R^{-T} per head leaves L_JAB unchanged."""
    for Hq, Hkv in ((2, 2), (4, 2)):
        desc, x, w = _tiny(Hq=Hq, Hkv=Hkv, dh=4, d=8)
        a = O.block_forward(x, w, desc)
        rng = np.random.default_rng(5)
        w2 = w.copy()
        r = Hq // Hkv
        for g in range(Hkv):
            R = rng.standard_normal((4, 4)) + 3 * np.eye(4)
            for h in range(g * r, (g + 1) * r):
                w2[h * 4:(h + 1) * 4] = R.T @ w[h * 4:(h + 1) * 4]           # Q_h -> Q_h R
            k0 = Hq * 4 + g * 4
            w2[k0:k0 + 4] = np.linalg.inv(R) @ w[k0:k0 + 4]                   # K_g -> K_g R^{-T}
        np.testing.assert_allclose(O.block_forward(x, w2, desc), a, atol=1e-11)


def test_scalar_head_toy_example_exact_zero_damage():
    """App. B, d_head = 1: delta_q = eps q with delta_k = -eps/(1+eps) k reproduces q k^T exactly,
    so the joint loss is zero although both matrices moved."""
    desc, x, w = _tiny(Hq=1, Hkv=1, dh=1, d=4, G=4)
    eps = 0.25
    w2 = w.copy()
    w2[0] = w[0] * (1 + eps)
    w2[1] = w[1] - eps / (1 + eps) * w[1]
    a, a2 = O.block_forward(x, w, desc), O.block_forward(x, w2, desc)
    np.testing.assert_allclose(a2, a, atol=1e-14)


def test_hessian_null_space_dimension_at_float_point():
    """Section 2.3: the per-head invariance gives H_L a null space of dimension >= n_head*d_head^2.

    At w*, H = 2 J^T J / n (Eq. 5 with lambda_KL = 0), so the null space is that of the Jacobian
    J = dA/dw, computed here by central differences on a block with more outputs than weights.
    """
    for Hq, dh in ((1, 2), (2, 2)):
        desc = _desc(3, Hq, Hq, dh, 3)
        rng = np.random.default_rng(11)
        x = rng.standard_normal((2, 16, 3))
        D = 3 * Hq * dh
        w = rng.standard_normal((D, 3)) * 0.7
        n_w = w.size
        J = np.empty((2 * 16 * Hq * dh, n_w))
        h = 1e-5
        for i in range(n_w):
            e = np.zeros(n_w)
            e[i] = h
            ap = O.block_forward(x, w + e.reshape(w.shape), desc)
            am = O.block_forward(x, w - e.reshape(w.shape), desc)
            J[:, i] = ((ap - am) / (2 * h)).ravel()
        sv = np.linalg.svd(J, compute_uv=False)
        null = int((sv < 1e-6 * sv[0]).sum())
        assert null >= Hq * dh * dh, (Hq, dh, sv)


# ------------------------------------------------------------------ loss (Section 2.2, Eq. 3)

def test_loss_zero_when_weights_on_grid():
    desc, x, _ = _tiny(rope=True)
    rng = np.random.default_rng(4)
    D, d = 16, 8
    q = rng.integers(-3, 4, size=(D, d))
    s = np.full((D, d // 4), 2.0 ** -4, dtype=np.float32)
    w = q * 2.0 ** -4
    r = O.jab_loss(x, w, s, 3, desc)
    assert r["loss"] == 0.0 and r["sse"] == 0.0
    g = O.jab_loss_and_grad(x, w, s, 3, desc)
    assert g["loss"] == 0.0 and not g["grad_s"].any()
    # the STE weight gradient vanishes identically at the float point (App. B, Fisher-coupling:
    # why a gradient score needs an off-grid probe)
    assert not g["grad_w_hat"].any()


def test_single_token_closed_form():
    """T = 1: softmax over one key is 1, so A = V; L = ||X (W_V_hat - W_V)^T||^2 / (B Hq d_h)
    mapped through the GQA head map, and the Q/K scale gradients are exactly zero."""
    desc, x, w = _tiny(T=1, Hq=4, Hkv=2, dh=4, rope=True)
    s = O.init_scales_absmax(w, 2, 4)
    r = O.jab_loss_and_grad(x, w, s, 2, desc, kappa=1.0)
    _, w_hat, _ = O.quantize(w, s, 2, 4)
    dv = (x[:, 0] @ (w_hat[24:32] - w[24:32]).T).reshape(-1, 2, 4)   # [B, Hkv, dh]
    sse = sum(((dv[:, h // 2]) ** 2).sum() for h in range(4))
    np.testing.assert_allclose(r["sse"], sse, rtol=1e-12)
    np.testing.assert_allclose(r["loss"], sse / (x.shape[0] * 4 * 4), rtol=1e-12)
    assert not r["grad_s"][:24].any()


def test_loss_quadratic_at_float_point():
    """Eq. 5: L_JAB is zero and stationary at w*, so L(w* + eps*Delta) / eps^2 tends to
    ||J_A Delta||^2 / n, with J_A Delta a central-difference directional derivative."""
    desc, x, w = _tiny(rope=True)
    rng = np.random.default_rng(6)
    delta = rng.standard_normal(w.shape) * 0.05
    a0 = O.block_forward(x, w, desc)
    n = a0.size
    ratios = []
    for eps in (1e-3, 1e-4):
        ratios.append(((O.block_forward(x, w + eps * delta, desc) - a0) ** 2).sum() / n / eps ** 2)
    h = 1e-6
    jvp = (O.block_forward(x, w + h * delta, desc) - O.block_forward(x, w - h * delta, desc)) / (2 * h)
    gn = (jvp ** 2).sum() / n
    np.testing.assert_allclose(ratios[1], gn, rtol=1e-3)
    np.testing.assert_allclose(ratios[0], ratios[1], rtol=3e-2)


def test_loss_shrinks_with_bits():
    """Finer grids shrink the error: L(b) strictly decreases over b = 2..8 on a random block."""
    desc, x, w = _tiny(T=8, rope=True, w_std=0.5)
    losses = [O.jab_loss(x, w, O.init_scales_absmax(w, b, 4), b, desc)["loss"] for b in (2, 3, 4, 5, 8)]
    assert all(l1 > l2 for l1, l2 in zip(losses, losses[1:])), losses


# ------------------------------------------------------------------ gradients (Eq. 13)

def _loss_at_w_hat(x, w_hat, desc, a_ref):
    return ((O.block_forward(x, w_hat, desc) - a_ref) ** 2).sum() / a_ref.size


@pytest.mark.parametrize("rope,Hq,Hkv", [(False, 2, 2), (True, 2, 1)])
def test_weight_gradient_matches_finite_differences(rope, Hq, Hkv):
    """STE weight gradient dL/dw_hat (Eq. 13, d w_hat / d w = 1) against central differences."""
    desc, x, w = _tiny(rope=rope, Hq=Hq, Hkv=Hkv, T=5)
    s = O.init_scales_absmax(w, 3, 4)
    g = O.jab_loss_and_grad(x, w, s, 3, desc, kappa=1.0)
    a_ref, w_hat = g["a_ref"], g["w_hat"]
    h = 1e-6
    rng = np.random.default_rng(7)
    idx = [tuple(i) for i in rng.integers(0, [w.shape[0], w.shape[1]], size=(24, 2))]
    for i in idx:
        wp, wm = w_hat.copy(), w_hat.copy()
        wp[i] += h
        wm[i] -= h
        fd = (_loss_at_w_hat(x, wp, desc, a_ref) - _loss_at_w_hat(x, wm, desc, a_ref)) / (2 * h)
        np.testing.assert_allclose(g["grad_w_hat"][i], fd, rtol=1e-5, atol=1e-11)


@pytest.mark.parametrize("bits", [2, 3])
def test_scale_gradient_matches_lsq_surrogate_finite_differences(bits):
    """LSQ rule (Eq. 13) against central differences of the frozen-code surrogate
    w_hat(s') = s' q + w (1 - s'/s) where |v| <= qmax, and s' sign(v) qmax elsewhere: its
    derivative at s' = s is exactly the rule, so FD of L(w_hat(s')) must equal grad_s (kappa=1)."""
    desc, x, w = _tiny(rope=True, T=5)
    G = 4
    s = O.init_scales_absmax(w, bits, G) * np.float32(0.8)
    g = O.jab_loss_and_grad(x, w, s, bits, desc, kappa=1.0)
    codes, w_hat, v = O.quantize(w, s, bits, G)
    qm = (1 << (bits - 1)) - 1
    inside = np.abs(v) <= qm
    a_ref = g["a_ref"]
    h = 1e-7
    for o in range(w.shape[0]):
        for gi in range(w.shape[1] // G):
            cols = slice(gi * G, (gi + 1) * G)

            def surrogate(sp):
                wh = w_hat.copy()
                qv = codes[o, cols].astype(np.float64)
                wv = w[o, cols]
                ins = inside[o, cols]
                wh[o, cols] = np.where(ins, sp * qv + wv * (1 - sp / float(s[o, gi])),
                                       sp * np.sign(v[o, cols]) * qm)
                return _loss_at_w_hat(x, wh, desc, a_ref)

            s0 = float(s[o, gi])
            fd = (surrogate(s0 + h) - surrogate(s0 - h)) / (2 * h)
            np.testing.assert_allclose(g["grad_s"][o, gi], fd, rtol=2e-5, atol=1e-12)


def _joint_at_w_hat(x, w_hat, desc, a_ref, P_teacher, lam):
    """MSE + lam * KL at given quantized weights, the KL from scipy's elementwise relative entropy."""
    special = pytest.importorskip("scipy.special")
    a_hat, parts = O.block_forward(x, w_hat, desc, return_parts=True)
    mse = ((a_hat - a_ref) ** 2).sum() / a_ref.size
    kl = special.rel_entr(P_teacher, parts["P"]).sum() / x.shape[0]
    return mse + lam * kl


@pytest.mark.parametrize("rope,Hq,Hkv,lam", [(False, 2, 2, 0.1), (True, 2, 1, 0.1),
                                             (True, 2, 1, 3e-4)])
def test_joint_weight_gradient_matches_finite_differences(rope, Hq, Hkv, lam):
    """dL/dw_hat of MSE + lam * KL (Eq. 3 with both terms, readings R3 and R18) against central
    differences; lam = 3e-4 puts the two terms' gradients at comparable size on this block."""
    desc, x, w = _tiny(rope=rope, Hq=Hq, Hkv=Hkv, T=5)
    s = O.init_scales_absmax(w, 2, 4)
    g = O.jab_loss_joint_and_grad(x, w, s, 2, desc, lam_kl=lam, kappa=1.0)
    a_ref, w_hat = g["a_ref"], g["w_hat"]
    _, teacher = O.block_forward(x, w, desc, return_parts=True)
    P = teacher["P"]
    np.testing.assert_allclose(g["loss"], _joint_at_w_hat(x, w_hat, desc, a_ref, P, lam), rtol=1e-12)
    h = 1e-6
    rng = np.random.default_rng(11)
    idx = [tuple(i) for i in rng.integers(0, [w.shape[0], w.shape[1]], size=(24, 2))]
    for i in idx:
        wp, wm = w_hat.copy(), w_hat.copy()
        wp[i] += h
        wm[i] -= h
        fd = (_joint_at_w_hat(x, wp, desc, a_ref, P, lam) -
              _joint_at_w_hat(x, wm, desc, a_ref, P, lam)) / (2 * h)
        np.testing.assert_allclose(g["grad_w_hat"][i], fd, rtol=1e-5, atol=1e-11)


def test_joint_scale_gradient_matches_lsq_surrogate_finite_differences():
    """The LSQ rule (Eq. 13) on the joint objective: central differences of the frozen-code
    surrogate (as for the MSE term) of MSE + 0.1 KL equal grad_s (kappa = 1)."""
    desc, x, w = _tiny(rope=True, T=5)
    G, bits, lam = 4, 2, 0.1
    s = O.init_scales_absmax(w, bits, G) * np.float32(0.8)
    g = O.jab_loss_joint_and_grad(x, w, s, bits, desc, lam_kl=lam, kappa=1.0)
    codes, w_hat, v = O.quantize(w, s, bits, G)
    inside = np.abs(v) <= 1
    a_ref = g["a_ref"]
    _, teacher = O.block_forward(x, w, desc, return_parts=True)
    h = 1e-7
    for o in range(0, w.shape[0], 3):
        for gi in range(w.shape[1] // G):
            cols = slice(gi * G, (gi + 1) * G)

            def surrogate(sp):
                wh = w_hat.copy()
                wh[o, cols] = np.where(inside[o, cols],
                                       sp * codes[o, cols] + w[o, cols] * (1 - sp / float(s[o, gi])),
                                       sp * np.sign(v[o, cols]))
                return _joint_at_w_hat(x, wh, desc, a_ref, teacher["P"], lam)

            s0 = float(s[o, gi])
            fd = (surrogate(s0 + h) - surrogate(s0 - h)) / (2 * h)
            np.testing.assert_allclose(g["grad_s"][o, gi], fd, rtol=2e-5, atol=1e-12)


def test_joint_gradient_reduces_to_the_mse_gradient_and_splits_into_its_terms():
    """lam = 0 gives the MSE term's loss and gradient; the KL value is kl_attention_term's; and the
    gradient is linear in lam (the KL term's gradient does not depend on lam)."""
    desc, x, w = _tiny(rope=True, T=6)
    s = O.init_scales_absmax(w, 3, 4)
    g0 = O.jab_loss_joint_and_grad(x, w, s, 3, desc, lam_kl=0.0)
    ref = O.jab_loss_and_grad(x, w, s, 3, desc, kappa=1.0)
    np.testing.assert_allclose(g0["loss"], ref["loss"], rtol=1e-13)
    np.testing.assert_allclose(g0["grad_s"], ref["grad_s"], rtol=1e-11, atol=1e-16)
    g1 = O.jab_loss_joint_and_grad(x, w, s, 3, desc, lam_kl=0.1)
    g2 = O.jab_loss_joint_and_grad(x, w, s, 3, desc, lam_kl=0.2)
    np.testing.assert_allclose(g1["kl"], O.kl_attention_term(x, w, s, 3, desc)["kl"], rtol=1e-13)
    np.testing.assert_allclose(g2["grad_s"] - g1["grad_s"], g1["grad_s"] - g0["grad_s"],
                               rtol=1e-9, atol=1e-15)
    assert np.abs(g1["grad_s"] - g0["grad_s"]).max() > 1e-3 * np.abs(g0["grad_s"]).max()


def test_kappa_is_a_pure_multiplier_and_default():
    desc, x, w = _tiny(rope=True)
    s = O.init_scales_absmax(w, 3, 4)
    g1 = O.jab_loss_and_grad(x, w, s, 3, desc, kappa=1.0)
    g2 = O.jab_loss_and_grad(x, w, s, 3, desc, kappa=0.0)
    np.testing.assert_allclose(g2["grad_s"], g1["grad_s"] / np.sqrt(4 * 3), rtol=1e-14)
    assert O.default_kappa(3, 128) == 1 / np.sqrt(128 * 3)


# ------------------------------------------------------------------ KL term of Eq. 3 (reading R18)

def _kl_case(seed=0, rope=True, bits=2, B=2, T=6):
    desc, x, w = _tiny(seed=seed, rope=rope, B=B, T=T)
    s = O.init_scales_absmax(w, bits, 4)
    return desc, x, w, s


@pytest.mark.parametrize("rope", [False, True])
def test_kl_term_matches_library_relative_entropy(rope):
    """sum(rel_entr(P, Q)) / B from scipy's elementwise relative entropy, per row and in total."""
    special = pytest.importorskip("scipy.special")
    desc, x, w, s = _kl_case(rope=rope)
    r = O.kl_attention_term(x, w, s, 2, desc)
    rows = special.rel_entr(r["P"], r["Q"]).sum(axis=3)
    np.testing.assert_allclose(r["kl_rows"], rows, rtol=1e-12, atol=1e-15)
    np.testing.assert_allclose(r["kl"], rows.sum() / x.shape[0], rtol=1e-12)
    assert r["kl"] > 0.0


def test_kl_row_logit_identity():
    """With log P = s^T - lse^T and log Q = s^S - lse^S on the visible keys, and rows of P summing to
    one: KL_row = sum_j P_j (s^T_j - s^S_j) + lse^S - lse^T (scores and lse taken from the teacher's
    and the student's own forward passes)."""
    desc, x, w, s = _kl_case(seed=3)
    r = O.kl_attention_term(x, w, s, 2, desc)
    _, w_hat, _ = O.quantize(w, s, 2, 4)
    _, tp = O.block_forward(x, w, desc, return_parts=True)
    _, sp = O.block_forward(x, w_hat, desc, return_parts=True)
    scale = 1.0 / np.sqrt(desc["head_dim"])
    B, T, Hq, _ = tp["q"].shape
    for b in range(B):
        for h in range(Hq):
            g = h // (Hq // desc["n_kv_heads"])
            st = tp["q"][b, :, h] @ tp["k"][b, :, g].T * scale
            ss = sp["q"][b, :, h] @ sp["k"][b, :, g].T * scale
            for t in range(T):
                p = tp["P"][b, h, t, : t + 1]
                kl = float(p @ (st[t, : t + 1] - ss[t, : t + 1])) + sp["lse"][b, h, t] - tp["lse"][b, h, t]
                np.testing.assert_allclose(r["kl_rows"][b, h, t], kl, rtol=1e-9, atol=1e-14)


def test_kl_zero_on_grid_and_for_a_single_token():
    desc, x, _ = _tiny(rope=True)
    rng = np.random.default_rng(5)
    w = rng.integers(-3, 4, size=(16, 8)) * 2.0 ** -4
    s = np.full((16, 2), 2.0 ** -4, dtype=np.float32)
    assert O.kl_attention_term(x, w, s, 3, desc)["kl"] == 0.0           # student = teacher
    desc1, x1, w1, s1 = _kl_case(T=1)
    r = O.kl_attention_term(x1, w1, s1, 2, desc1)                          # one key: P = Q = 1
    assert r["kl"] == 0.0 and not r["kl_rows"].any()


def test_kl_nonnegative_rows_and_batchmean():
    """Gibbs' inequality row by row; batchmean: repeating the batch leaves the value unchanged."""
    for seed in range(4):
        desc, x, w, s = _kl_case(seed=seed)
        r = O.kl_attention_term(x, w, s, 2, desc)
        assert (r["kl_rows"] >= -1e-15).all()
        r2 = O.kl_attention_term(np.concatenate([x, x]), w, s, 2, desc)
        np.testing.assert_allclose(r2["kl"], r["kl"], rtol=1e-12)
        np.testing.assert_allclose(r2["kl_rows"].sum(), 2 * r["kl_rows"].sum(), rtol=1e-12)


def test_joint_loss_is_mse_plus_weighted_kl():
    desc, x, w, s = _kl_case(seed=2)
    j0 = O.jab_loss_joint(x, w, s, 2, desc, lam_kl=0.0)
    assert j0["loss"] == O.jab_loss(x, w, s, 2, desc)["loss"]
    j = O.jab_loss_joint(x, w, s, 2, desc)                      # lambda_KL = 0.1 (Section 3)
    np.testing.assert_allclose(j["loss"], j["mse"] + 0.1 * j["kl"], rtol=1e-15)


# ------------------------------------------------------------------ sensitivity (Section 2.4, R19)

@pytest.mark.parametrize("rope,Hq,Hkv", [(False, 2, 1), (True, 2, 2), (True, 4, 2)])
def test_block_jvp_matches_central_differences(rope, Hq, Hkv):
    desc, x, w = _tiny(seed=7, rope=rope, Hq=Hq, Hkv=Hkv)
    V = np.random.default_rng(8).standard_normal(w.shape)
    h = 1e-6
    fd = (O.block_forward(x, w + h * V, desc) - O.block_forward(x, w - h * V, desc)) / (2 * h)
    np.testing.assert_allclose(O.block_jvp(x, w, V, desc), fd, rtol=1e-6, atol=1e-9)


def test_gn_quadratic_form_is_the_second_difference_of_the_loss():
    """At the float point L(w* + eps v) = eps^2 v^T H v / 2 + O(eps^3) (L and its gradient vanish
    there), so the symmetric second difference (L(eps) + L(-eps)) / eps^2 gives v^T H v."""
    desc, x, w = _tiny(seed=9, rope=True)
    a_ref = O.block_forward(x, w, desc)
    V = np.random.default_rng(10).standard_normal(w.shape)

    def loss(e):
        return float(((O.block_forward(x, w + e * V, desc) - a_ref) ** 2).mean())

    eps = 1e-3
    np.testing.assert_allclose((loss(eps) + loss(-eps)) / eps ** 2, O.gn_quadratic_form(x, w, V, desc),
                               rtol=1e-4)


def test_hutchinson_trace_matches_the_exact_trace():
    """Exact Tr(H) = 2 sum_k ||J e_k||^2 / n from a central-difference Jacobian; the estimator over
    m Rademacher probes lies within 5 standard errors, sqrt(2 sum_{i != j} H_ij^2 / m)."""
    desc = _desc(4, 1, 1, 2, 4, rope=True)
    rng = np.random.default_rng(12)
    x = rng.standard_normal((1, 6, 4))
    w = rng.standard_normal((6, 4)) * 0.6
    n_w = w.size
    J = np.empty((6 * 2, n_w))
    h = 1e-6
    for i in range(n_w):
        e = np.zeros(n_w)
        e[i] = h
        J[:, i] = ((O.block_forward(x, w + e.reshape(w.shape), desc) -
                    O.block_forward(x, w - e.reshape(w.shape), desc)) / (2 * h)).ravel()
    H = 2.0 * J.T @ J / J.shape[0]
    m = 3000
    probes = rng.choice([-1.0, 1.0], size=(m,) + w.shape)
    est = O.hutchinson_trace(x, w, desc, probes)
    off = H - np.diag(np.diag(H))
    se = np.sqrt(2.0 * (off ** 2).sum() / m)
    assert abs(est - np.trace(H)) <= 5 * se, (est, np.trace(H), se)
    # one probe direction against the explicit quadratic form
    np.testing.assert_allclose(O.gn_quadratic_form(x, w, probes[0], desc),
                               probes[0].ravel() @ H @ probes[0].ravel(), rtol=1e-6)


def test_gn_quadratic_form_vanishes_on_the_query_key_scaling_direction():
    """W_Q (1 + e), W_K / (1 + e) leaves A unchanged (RoPE commutes with the scalar), so its tangent
    (W_Q, -W_K, 0) is in the null space of J_A and of H (Section 2.3)."""
    desc, x, w = _tiny(seed=13, rope=True)
    nq = desc["n_q_heads"] * desc["head_dim"]
    nk = desc["n_kv_heads"] * desc["head_dim"]
    V = np.zeros_like(w)
    V[:nq] = w[:nq]
    V[nq:nq + nk] = -w[nq:nq + nk]
    ref = O.gn_quadratic_form(x, w, np.random.default_rng(14).standard_normal(w.shape), desc)
    assert O.gn_quadratic_form(x, w, V, desc) <= 1e-12 * ref


def test_omega_scores_vanish_on_the_grid_and_scale_with_depth():
    desc, _, _ = _tiny()
    rng = np.random.default_rng(15)
    w = rng.integers(-3, 4, size=(16, 8)) * 2.0 ** -4
    s = np.full((16, 2), 2.0 ** -4, dtype=np.float32)
    assert O.omega_scores(2.5, w, s, 3, 4, layers_after=3) == (0.0, 0.0)
    w2 = w + rng.standard_normal(w.shape) * 2.0 ** -7
    c1, c2 = O.omega_scores(2.5, w2, s, 3, 4, layers_after=3)
    assert c1 > 0 and c2 == 3 * c1


def test_splitmix64_published_outputs_and_probe_signs():
    """The probes' generator reproduces SplitMix64's published first outputs; probe entries take
    their sign from the top bit, probe i starting at counter i * size; the signs are balanced."""
    with open(os.path.join(GOLDEN, "splitmix64.json")) as f:
        fx = json.load(f)
    want = [int(h, 16) for h in fx["outputs_hex"]]
    assert [int(v) for v in O.splitmix64(fx["seed"], [0, 1, 2])] == want
    assert O.rademacher_probe(0, 0, (1, 3)).tolist() == [[-1.0 if v >> 63 else 1.0 for v in want]]
    p1 = O.rademacher_probe(0, 1, (1, 3))            # probe 1 starts at counter 3
    assert p1[0, 0] == (-1.0 if int(O.splitmix64(0, [3])[0]) >> 63 else 1.0)
    big = O.rademacher_probe(7, 2, (200, 500))
    assert set(np.unique(big)) == {-1.0, 1.0} and abs(big.mean()) < 5 / np.sqrt(big.size)


def test_omega_scores_hand_worked():
    """Eq. 6 on one row worked by hand. b = 3 (qmax = 3), one group of 5, s = 1/2:
    w      = 0.375, -0.6875, 1.25, 0.0625, 2.0
    w / s  = 0.75,  -1.375,  2.5,  0.125,  4.0
    q      = 1,     -1,      2,    0,      3      (2.5 -> 2 half to even; 4 clamps to qmax)
    Q(w)   = 0.5,   -0.5,    1.0,  0.0,    1.5
    Q(w)-w = 0.125, 0.1875, -0.25, -0.0625, -0.5
    ||Q(w) - W||_F^2 = 1/64 + 9/256 + 1/16 + 1/256 + 1/4 = 0.3671875.
    With Tr(H) = 2: C1 = 0.734375; with L - i = 3 layers after it: C2 = 2.203125."""
    w = np.array([[0.375, -0.6875, 1.25, 0.0625, 2.0]])
    s = np.array([[0.5]], dtype=np.float32)
    c1, c2 = O.omega_scores(2.0, w, s, 3, 5, layers_after=3)
    assert c1 == 0.734375 and c2 == 2.203125


# ------------------------------------------------------------------ allocation (Eq. 7, App. B, R20)

def test_allocation_hand_worked_example():
    """Widths (2, 4, 8), 10 weights per layer, 4 bits on average (80 bits). From (8, 8), 160 bits:
    layer 0 8 -> 4 costs (2 - 1) / 40 = 0.025 per bit against (3 - 0.5) / 40 = 0.0625 for layer 1,
    then layer 1 8 -> 4 (0.0625 < (5 - 2) / 20 = 0.15) meets 80 bits; no upgrade fits."""
    om = [[5.0, 2.0, 1.0], [9.0, 3.0, 0.5]]
    for method in ("greedy", "pareto"):
        assert O.allocate_bits(om, [2, 4, 8], [10, 10], 4.0, method) == [4, 4]
    # 5 bits on average (100 bits): the leftover 20 bits cannot buy an 8-bit layer (+40)
    assert O.allocate_bits(om, [2, 4, 8], [10, 10], 5.0) == [4, 4]
    # 6 bits (120): after layer 0's first step the budget holds at (4, 8)
    assert O.allocate_bits(om, [2, 4, 8], [10, 10], 6.0) == [4, 8]


def test_allocation_extremes_and_infeasible_budget():
    rng = np.random.default_rng(20)
    om = np.sort(rng.random((5, 4)), axis=1)[:, ::-1]
    n = rng.integers(1, 100, size=5)
    assert O.allocate_bits(om, [2, 3, 4, 8], n, 8.0) == [8] * 5
    assert O.allocate_bits(om, [2, 3, 4, 8], n, 2.0) == [2] * 5
    with pytest.raises(ValueError):
        O.allocate_bits(om, [2, 3, 4, 8], n, 1.99)


def test_greedy_is_optimal_for_convex_scores_with_unit_steps():
    """Marginal analysis: for separable convex, decreasing scores and equal cost steps (widths one
    bit apart, one weight per layer), the greedy walk reaches the exhaustive-search optimum."""
    import itertools
    rng = np.random.default_rng(21)
    widths = [2, 3, 4, 5, 6]
    for _ in range(40):
        L = int(rng.integers(2, 5))
        steps = np.sort(rng.random((L, len(widths) - 1)), axis=1)[:, ::-1]   # shrinking decrements
        om = np.concatenate([np.zeros((L, 1)), -np.cumsum(steps, axis=1)], axis=1) + 10.0
        budget = int(rng.integers(2 * L, 6 * L + 1))
        got = O.allocate_bits(om, widths, [1] * L, budget / L)
        best = min(sum(om[i][widths.index(b)] for i, b in enumerate(c))
                   for c in itertools.product(widths, repeat=L) if sum(c) <= budget)
        assert sum(got) <= budget
        np.testing.assert_allclose(sum(om[i][widths.index(b)] for i, b in enumerate(got)), best,
                                   rtol=1e-12)


def test_greedy_result_is_feasible_and_admits_no_improving_upgrade():
    rng = np.random.default_rng(22)
    widths = [2, 3, 4, 8, 16]
    for _ in range(50):
        L = int(rng.integers(1, 7))
        om = rng.random((L, len(widths))) * rng.random()
        n = rng.integers(1, 50, size=L)
        avg = float(rng.uniform(2.0, 16.0))
        for method in ("greedy", "pareto"):
            got = O.allocate_bits(om, widths, n, avg, method)
            cost = sum(int(n[i]) * b for i, b in enumerate(got))
            assert cost <= avg * n.sum()
            if method == "greedy":
                for i, b in enumerate(got):      # every single upgrade either does not fit or does not help
                    k = widths.index(b)
                    if k + 1 < len(widths):
                        fits = cost + int(n[i]) * (widths[k + 1] - b) <= avg * n.sum()
                        assert not (fits and om[i][k + 1] < om[i][k])


def test_pareto_frontier_keeps_exactly_the_non_dominated_points():
    rng = np.random.default_rng(23)
    for _ in range(100):
        K = int(rng.integers(1, 7))
        costs = np.sort(rng.choice(100, size=K, replace=False))
        oms = rng.integers(0, 5, size=K).astype(float)                 # ties on purpose
        kept = O.pareto_frontier(costs, oms)
        brute = [k for k in range(K)
                 if not any(j != k and costs[j] <= costs[k] and oms[j] <= oms[k] for j in range(K))]
        assert kept == brute
