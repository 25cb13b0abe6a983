"""Float64 CPU oracle for the joint attention-block loss L_JAB and its STE/LSQ scale gradient.

TEST INFRASTRUCTURE ONLY. Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline /
reference legs may import or run this module. The product path (the C-ABI library and its
Python binding) never imports it, and it never imports the product path.

Plain, slow, obviously correct: numpy in float64, one step of the paper per function, no
blocking, fusion or reordering beyond what the definitions state. numpy's matmul is used as a
library primitive for the projection and the attention products.

What it computes (paper: Section 2.1 Eq. 2, Section 2.2 Eq. 3, App. B "Effective weight of the
KL term", App. B "Joint STE fine-tuning" Eq. 13, App. C "Models and scope"):

  1. quantizer          v = fl32(w / s), q = clip(round_half_even(v), -qmax, qmax), w_hat = q*s
  2. joint projection   [Q | K | V] = X W^T  (W = [W_Q; W_K; W_V] in nn.Linear layout)
  3. RoPE               rotate-half on every Q and K head, positions 0..T-1 per sequence
  4. attention          A = softmax(Q K^T / sqrt(d_h) + M) V, causal M, GQA head map
  5. loss               L = ||A(X; W) - A(X; w_hat)||_F^2 / (B * T * Hq * d_h)   (MSE term)
  6. backward           dL/dw_hat by the attention VJP, then the LSQ rule for dL/ds.

Readings of points the paper leaves open (each is stated where it is used):
  R1  w/s is the IEEE fp32 quotient and round() is round-half-to-even.
  R2  the code range is symmetric [-qmax, qmax], qmax = 2^(b-1) - 1.
  R3  the MSE term is an element-wise mean over B*T*(Hq*d_h) entries; SSE is also returned.
  R4  the hot path's loss is the MSE term (lambda_KL = 0); jab_loss_joint and
      jab_loss_joint_and_grad add lambda_KL times the KL term (R18) and its gradient.
  R5  the LSQ branch tests |v| <= qmax on the unrounded quotient v.
  R6  n_w in (n_w * qmax)^(-1/2) is the group size G; it is exposed as kappa.
  R7  RoPE is the rotate-half convention with inv_freq_j = theta^(-2j/d_h).
  R8  GQA: query head h reads key/value head floor(h / (Hq / Hkv)).
  R9  an all-zero group gets scale 1 at absmax init (any positive scale gives code 0).
  R18 the KL term of Eq. 3 is D_KL(P || Q(w)) with the implemented
      batchmean convention: the sum over sequences, query heads, query rows and keys of
      P log(P / Q), divided by B; P is the teacher's post-softmax map, Q the student's; masked
      entries have P = Q = 0 and contribute nothing; lambda_KL defaults to 0.1 (Section 3).
  R19 the sensitivity criterion (Section 2.4, Eq. 5-6) is taken for the
      MSE term as normalised in R3 (lambda_KL = 0): at the float point H = 2 J_A^T J_A / n with
      n = B*T*Hq*d_h, so v^T H v = 2 ||J_A v||^2 / n; the Rademacher probes are inputs.
  R21 the flip rate of Eq. 15 counts the grid positions (the clamped codes of Eq. 2, i.e. the
      deployed values) that differ between two quantizations of the same weights, over d' = the
      number of weights compared.
  R20 allocation (Section 2.4, Eq. 7; App. B "Allocators"): layer i at width b costs n_i * b bits and
      the budget is avg_bits * sum_i n_i (the parameter-weighted budget of Eq. 8); each greedy step moves one layer to the adjacent width of
      its candidate list; the step ratio is dOmega / dcost in float64; ties go to the lowest layer
      index; after the budget is met, upgrades are applied while one fits and lowers sum Omega
      (best gain per bit first). The Pareto variant walks each layer's non-dominated points only.
"""
from __future__ import annotations

import numpy as np

__all__ = [
    "qmax_of", "expand_groups", "fp32_quotient", "quantize", "init_scales_absmax",
    "init_scales_minmse", "project", "rope_tables", "apply_rope", "apply_rope_transpose",
    "split_heads", "causal_gqa_attention", "block_forward", "jab_loss", "attention_vjp",
    "jab_loss_and_grad", "lsq_factor", "default_kappa", "kl_attention_term", "jab_loss_joint",
    "attention_jvp", "block_jvp", "gn_quadratic_form", "hutchinson_trace", "omega_scores",
    "pareto_frontier", "allocate_bits", "flip_count", "splitmix64", "rademacher_probe",
]


# --------------------------------------------------------------------------------------------
# 1. Quantizer (Section 2.1, Eq. 2)
# --------------------------------------------------------------------------------------------

def qmax_of(bits: int) -> int:
    """qmax = 2^(b-1) - 1 (Eq. 2). b=2 gives the symmetric code set {-1, 0, 1} (reading R2)."""
    if bits < 2:
        raise ValueError("bits must be >= 2")
    return (1 << (bits - 1)) - 1


def expand_groups(s: np.ndarray, group_size: int) -> np.ndarray:
    """One scale per (output row, group): s[o, g] applies to columns g*G .. g*G+G-1 (Section 2.1)."""
    return np.repeat(np.asarray(s), group_size, axis=1)


def fp32_quotient(w: np.ndarray, s_full: np.ndarray) -> np.ndarray:
    """v = w / s as an IEEE single-precision quotient (reading R1), returned as float64.

    w holds bf16 values and s fp32 values; both convert to float32 exactly.
    """
    w32 = np.asarray(w, dtype=np.float32)
    s32 = np.asarray(s_full, dtype=np.float32)
    return (w32 / s32).astype(np.float64)


def quantize(w: np.ndarray, s: np.ndarray, bits: int, group_size: int):
    """Eq. 2: Q(w) = clip(round(w/s), -qmax, qmax) * s with a per-(row, group) scale.

    Returns (codes int8, w_hat float64, v float64). w_hat = q * s is exact in float64
    (|q| < 2^7 times a 24-bit significand).
    """
    w = np.asarray(w, dtype=np.float64)
    s = np.asarray(s, dtype=np.float64)
    if not np.all(np.isfinite(s)) or np.any(s <= 0):
        raise ValueError("scales must be finite and > 0")
    qm = qmax_of(bits)
    s_full = expand_groups(s, group_size)
    v = fp32_quotient(w, s_full)
    q = np.clip(np.rint(v), -qm, qm)          # np.rint rounds half to even
    w_hat = q * s_full
    return q.astype(np.int8), w_hat, v


def flip_count(codes_a: np.ndarray, codes_b: np.ndarray) -> int:
    """Eq. 15 numerator: the number of positions whose grid position differs between two code
    arrays of the same weights (reading R21); the flip rate is this count over their size."""
    a = np.asarray(codes_a).ravel()
    b = np.asarray(codes_b).ravel()
    if a.shape != b.shape:
        raise ValueError("code arrays differ in size")
    return int(np.count_nonzero(a != b))


def init_scales_absmax(w: np.ndarray, bits: int, group_size: int) -> np.ndarray:
    """Starting scale max_{i in g} |w[o, i]| / qmax per group, as an fp32 quotient (reading R9)."""
    w = np.asarray(w, dtype=np.float64)
    D, d = w.shape
    amax = np.abs(w).reshape(D, d // group_size, group_size).max(axis=2)
    s = (amax.astype(np.float32) / np.float32(qmax_of(bits))).astype(np.float32)
    s[amax == 0] = np.float32(1.0)
    return s


def init_scales_minmse(w: np.ndarray, bits: int, group_size: int, n_grid: int = 80) -> np.ndarray:
    """Per-group min-MSE grid search over shrunken absmax scales (the warm-start scales).

    Candidates s_k = fl32(s_0 * (100 - k) / 100) for k = 0 .. n_grid-1 (product and quotient
    in float64, then one rounding to fp32); the chosen scale minimises sum_{i in g}
    (Q(w_i; s_k) - w_i)^2, ties going to the smallest k.
    """
    w = np.asarray(w, dtype=np.float64)
    D, d = w.shape
    ng = d // group_size
    s0 = init_scales_absmax(w, bits, group_size).astype(np.float64)
    best_err = np.full((D, ng), np.inf)
    best_s = s0.astype(np.float32).copy()
    qm = qmax_of(bits)
    wg = w.reshape(D, ng, group_size)
    for k in range(n_grid):
        sk = (s0 * (100 - k) / 100.0).astype(np.float32)
        v = (wg.astype(np.float32) / sk[:, :, None]).astype(np.float64)
        q = np.clip(np.rint(v), -qm, qm)
        err = ((q * sk[:, :, None].astype(np.float64) - wg) ** 2).sum(axis=2)
        better = err < best_err
        best_err = np.where(better, err, best_err)
        best_s = np.where(better, sk, best_s)
    return best_s.astype(np.float32)


# --------------------------------------------------------------------------------------------
# 2-4. Block forward: projection, RoPE, causal GQA attention (Section 2.1; App. C)
# --------------------------------------------------------------------------------------------

def project(x: np.ndarray, w: np.ndarray) -> np.ndarray:
    """Joint projection [Q | K | V] = X W^T with W in nn.Linear layout [D, d] (Section 2.1)."""
    x = np.asarray(x, dtype=np.float64)
    return x @ np.asarray(w, dtype=np.float64).T


def rope_tables(T: int, head_dim: int, theta: float):
    """cos/sin [T, d_h/2] of phi = t * theta^(-2j/d_h) (reading R7)."""
    j = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / head_dim)
    phi = np.arange(T, dtype=np.float64)[:, None] * inv_freq[None, :]
    return np.cos(phi), np.sin(phi)


def apply_rope(x: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Rotate-half RoPE on x [B, T, H, d_h]:  x'_j = x_j cos - x_{j+h} sin,
    x'_{j+h} = x_{j+h} cos + x_j sin, with h = d_h/2 and the angle of pair j at position t."""
    h = x.shape[-1] // 2
    c = cos[None, :, None, :]
    s = sin[None, :, None, :]
    x1, x2 = x[..., :h], x[..., h:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def apply_rope_transpose(g: np.ndarray, cos: np.ndarray, sin: np.ndarray) -> np.ndarray:
    """Transpose (= inverse) of the RoPE rotation, applied to gradients."""
    h = g.shape[-1] // 2
    c = cos[None, :, None, :]
    s = sin[None, :, None, :]
    g1, g2 = g[..., :h], g[..., h:]
    return np.concatenate([g1 * c + g2 * s, g2 * c - g1 * s], axis=-1)


def split_heads(qkv: np.ndarray, n_q_heads: int, n_kv_heads: int, head_dim: int):
    """[B, T, D] -> Q [B,T,Hq,d_h], K [B,T,Hkv,d_h], V [B,T,Hkv,d_h] (rows Q, then K, then V)."""
    B, T, _ = qkv.shape
    nq = n_q_heads * head_dim
    nk = n_kv_heads * head_dim
    q = qkv[:, :, :nq].reshape(B, T, n_q_heads, head_dim)
    k = qkv[:, :, nq:nq + nk].reshape(B, T, n_kv_heads, head_dim)
    v = qkv[:, :, nq + nk:nq + 2 * nk].reshape(B, T, n_kv_heads, head_dim)
    return q, k, v


def _kv_head(h: int, n_q_heads: int, n_kv_heads: int) -> int:
    """GQA head map (reading R8)."""
    return h // (n_q_heads // n_kv_heads)


def causal_gqa_attention(q, k, v, scale: float, return_p: bool = False):
    """A = softmax(Q K^T * scale + M) V per (sequence, query head), causal mask M (Section 2.1).

    q [B,T,Hq,d_h], k/v [B,T,Hkv,d_h] -> O [B,T,Hq,d_h]; optionally P [B,Hq,T,T] and the
    row log-sum-exp [B,Hq,T] of the scaled scores.
    """
    B, T, Hq, dh = q.shape
    Hkv = k.shape[2]
    mask = np.triu(np.ones((T, T), dtype=bool), k=1)      # j > t is masked
    out = np.empty((B, T, Hq, dh))
    P_all = np.empty((B, Hq, T, T)) if return_p else None
    lse = np.empty((B, Hq, T))
    for b in range(B):
        for h in range(Hq):
            g = _kv_head(h, Hq, Hkv)
            S = (q[b, :, h, :] @ k[b, :, g, :].T) * scale
            S = np.where(mask, -np.inf, S)
            m = S.max(axis=1, keepdims=True)
            E = np.exp(S - m)
            Z = E.sum(axis=1, keepdims=True)
            P = E / Z
            out[b, :, h, :] = P @ v[b, :, g, :]
            lse[b, h, :] = (m + np.log(Z))[:, 0]
            if return_p:
                P_all[b, h] = P
    return out, P_all, lse


def _softmax_scale(desc) -> float:
    sc = float(desc.get("softmax_scale", 0.0) or 0.0)
    return sc if sc > 0 else 1.0 / np.sqrt(desc["head_dim"])


def block_forward(x: np.ndarray, w: np.ndarray, desc: dict, return_parts: bool = False):
    """Attention output A(X; W) [B, T, Hq*d_h] of one block (merged heads, pre-o_proj)."""
    B, T, _ = x.shape
    Hq, Hkv, dh = desc["n_q_heads"], desc["n_kv_heads"], desc["head_dim"]
    qkv = project(x, w)
    q, k, v = split_heads(qkv, Hq, Hkv, dh)
    if desc.get("use_rope", False):
        cos, sin = rope_tables(T, dh, float(desc.get("rope_theta", 10000.0)))
        q = apply_rope(q, cos, sin)
        k = apply_rope(k, cos, sin)
    o, P, lse = causal_gqa_attention(q, k, v, _softmax_scale(desc), return_p=return_parts)
    a = o.reshape(B, T, Hq * dh)
    if return_parts:
        return a, dict(q=q, k=k, v=v, o=o, P=P, lse=lse)
    return a


# --------------------------------------------------------------------------------------------
# 5. Loss (Section 2.2, Eq. 3, MSE term; App. B "Effective weight of the KL term")
# --------------------------------------------------------------------------------------------

def jab_loss(x, w, s, bits: int, desc: dict, a_ref=None):
    """L_JAB MSE term for one candidate (reading R3, R4).

    a_ref is the teacher output A(X; W) with the float (bf16) weights; it is computed here when
    not given. Returns dict(loss, sse, sse_parts [B, Hq], codes, w_hat).
    """
    G = desc["group_size"]
    codes, w_hat, _ = quantize(w, s, bits, G)
    if a_ref is None:
        a_ref = block_forward(x, w, desc)
    a_hat = block_forward(x, w_hat, desc)
    B, T, _ = a_ref.shape
    Hq, dh = desc["n_q_heads"], desc["head_dim"]
    err = (a_hat - a_ref).reshape(B, T, Hq, dh)
    sse_parts = (err ** 2).sum(axis=(1, 3))
    sse = float(sse_parts.sum())
    return dict(loss=sse / (B * T * Hq * dh), sse=sse, sse_parts=sse_parts, codes=codes,
                w_hat=w_hat, a_ref=a_ref, a_hat=a_hat)


def kl_attention_term(x, w, s, bits: int, desc: dict):
    """D_KL(P || Q(w)), the second term of Eq. 3, batchmean as implemented (reading R18; App. B
    "Effective weight of the KL term"). P and Q are the post-softmax maps of the block with the
    float and with the quantized weights. Returns dict(kl, kl_rows [B, Hq, T], P, Q).
    """
    G = desc["group_size"]
    _, w_hat, _ = quantize(w, s, bits, G)
    _, teacher = block_forward(x, w, desc, return_parts=True)
    _, student = block_forward(x, w_hat, desc, return_parts=True)
    P, Q = teacher["P"], student["P"]
    with np.errstate(divide="ignore", invalid="ignore"):
        terms = np.where(P > 0, P * (np.log(P) - np.log(Q)), 0.0)   # 0 log 0 = 0 on masked keys
    kl_rows = terms.sum(axis=3)
    B = x.shape[0]
    return dict(kl=float(kl_rows.sum()) / B, kl_rows=kl_rows, P=P, Q=Q)


def jab_loss_joint(x, w, s, bits: int, desc: dict, lam_kl: float = 0.1):
    """Eq. 3 with both terms as implemented: the MSE mean (reading R3) plus lam_kl times the KL
    batchmean (reading R18). Returns dict(loss, mse, kl)."""
    mse = jab_loss(x, w, s, bits, desc)["loss"]
    kl = kl_attention_term(x, w, s, bits, desc)["kl"]
    return dict(loss=mse + lam_kl * kl, mse=mse, kl=kl)


# --------------------------------------------------------------------------------------------
# 6. Backward: attention VJP, STE on w_hat, LSQ rule on s (App. B "Joint STE fine-tuning", Eq. 13)
# --------------------------------------------------------------------------------------------

def attention_vjp(q, k, v, P, dO, scale: float, dS_extra=None):
    """Vector-Jacobian product of causal GQA attention.

    dV = P^T dO, dP = dO V^T, dS = P * (dP - rowsum(dP * P)), dQ = dS K * scale,
    dK = dS^T Q * scale; key/value gradients are summed over the query heads of a group.
    dS_extra [B, Hq, T, T] (optional) is a gradient of the loss with respect to the scaled scores
    S = Q K^T * scale that does not pass through O (the KL term of Eq. 3); it is added to dS.
    """
    B, T, Hq, dh = q.shape
    Hkv = k.shape[2]
    dq = np.zeros_like(q)
    dk = np.zeros_like(k)
    dv = np.zeros_like(v)
    for b in range(B):
        for h in range(Hq):
            g = _kv_head(h, Hq, Hkv)
            Ph = P[b, h]
            dOh = dO[b, :, h, :]
            dv[b, :, g, :] += Ph.T @ dOh
            dP = dOh @ v[b, :, g, :].T
            dS = Ph * (dP - (dP * Ph).sum(axis=1, keepdims=True))
            if dS_extra is not None:
                dS = dS + dS_extra[b, h]
            dq[b, :, h, :] = (dS @ k[b, :, g, :]) * scale
            dk[b, :, g, :] += (dS.T @ q[b, :, h, :]) * scale
    return dq, dk, dv


def lsq_factor(v: np.ndarray, bits: int) -> np.ndarray:
    """Eq. 13: d w_hat / d s = q - v if |v| <= qmax, else sign(v) * qmax (reading R5)."""
    qm = qmax_of(bits)
    q = np.clip(np.rint(v), -qm, qm)
    return np.where(np.abs(v) <= qm, q - v, np.sign(v) * qm)


def default_kappa(bits: int, group_size: int) -> float:
    """LSQ gradient scale (n_w * qmax)^(-1/2) with n_w = G (reading R6)."""
    return 1.0 / np.sqrt(group_size * qmax_of(bits))


def jab_loss_and_grad(x, w, s, bits: int, desc: dict, a_ref=None, kappa: float = 1.0):
    """L_JAB and its gradient w.r.t. the per-group scales (STE on weights, LSQ on scales).

    Returns dict(loss, sse, grad_s [D, d/G] = kappa * sum_{i in g} dL/dw_hat[o,i] * r[o,i],
    grad_w_hat [D, d] = dL/dw_hat (the STE weight gradient, d w_hat / d w = 1)).
    kappa <= 0 selects default_kappa(bits, G).
    """
    x = np.asarray(x, dtype=np.float64)
    G = desc["group_size"]
    Hq, Hkv, dh = desc["n_q_heads"], desc["n_kv_heads"], desc["head_dim"]
    B, T, d = x.shape
    codes, w_hat, v = quantize(w, s, bits, G)
    if a_ref is None:
        a_ref = block_forward(x, w, desc)
    a_hat, parts = block_forward(x, w_hat, desc, return_parts=True)
    n_el = B * T * Hq * dh
    diff = a_hat - a_ref
    sse = float((diff ** 2).sum())
    dO = (2.0 / n_el) * diff.reshape(B, T, Hq, dh)
    dq, dk, dv = attention_vjp(parts["q"], parts["k"], parts["v"], parts["P"], dO,
                               _softmax_scale(desc))
    if desc.get("use_rope", False):
        cos, sin = rope_tables(T, dh, float(desc.get("rope_theta", 10000.0)))
        dq = apply_rope_transpose(dq, cos, sin)
        dk = apply_rope_transpose(dk, cos, sin)
    dqkv = np.concatenate([dq.reshape(B, T, Hq * dh), dk.reshape(B, T, Hkv * dh),
                           dv.reshape(B, T, Hkv * dh)], axis=2)
    grad_w_hat = dqkv.reshape(B * T, -1).T @ x.reshape(B * T, d)      # [D, d]
    r = lsq_factor(v, bits)
    if kappa is None or kappa <= 0:
        kappa = default_kappa(bits, G)
    D = grad_w_hat.shape[0]
    grad_s = kappa * (grad_w_hat * r).reshape(D, d // G, G).sum(axis=2)
    return dict(loss=sse / n_el, sse=sse, grad_s=grad_s, grad_w_hat=grad_w_hat, codes=codes,
                w_hat=w_hat, a_ref=a_ref, a_hat=a_hat, lse=parts["lse"])


def jab_loss_joint_and_grad(x, w, s, bits: int, desc: dict, lam_kl: float = 0.1, kappa: float = 1.0):
    """Eq. 3 with both terms (readings R3, R18) and its STE / LSQ gradient w.r.t. the scales.

    L = MSE + lam_kl * KL with KL = sum over (sequence, query head, query row) of
    D_KL(P_row || Q_row) / B, P the teacher's map and Q the student's. Q_row = softmax(s_row) of the
    student's scaled scores s = Q K^T * scale, so d KL_row / d s_row = Q_row - P_row (the gradient
    of log-sum-exp minus the P-weighted scores); the KL term reaches the weights only through the
    student's scores, and adds (lam_kl / B) (Q - P) to the score gradient of the MSE term's
    attention VJP. Then the transpose of RoPE, dL/dw_hat = dQKV^T X and the LSQ rule (Eq. 13) as in
    jab_loss_and_grad. Returns dict(loss, mse, kl, grad_s, grad_w_hat).
    """
    x = np.asarray(x, dtype=np.float64)
    G = desc["group_size"]
    Hq, Hkv, dh = desc["n_q_heads"], desc["n_kv_heads"], desc["head_dim"]
    B, T, d = x.shape
    codes, w_hat, v = quantize(w, s, bits, G)
    a_ref, teacher = block_forward(x, w, desc, return_parts=True)
    a_hat, student = block_forward(x, w_hat, desc, return_parts=True)
    n_el = B * T * Hq * dh
    diff = a_hat - a_ref
    mse = float((diff ** 2).sum()) / n_el
    P, Qs = teacher["P"], student["P"]
    with np.errstate(divide="ignore", invalid="ignore"):
        kl = float(np.where(P > 0, P * (np.log(P) - np.log(Qs)), 0.0).sum()) / B
    dO = (2.0 / n_el) * diff.reshape(B, T, Hq, dh)
    dS_kl = (lam_kl / B) * (Qs - P)
    dq, dk, dv = attention_vjp(student["q"], student["k"], student["v"], Qs, dO,
                               _softmax_scale(desc), dS_extra=dS_kl)
    if desc.get("use_rope", False):
        cos, sin = rope_tables(T, dh, float(desc.get("rope_theta", 10000.0)))
        dq = apply_rope_transpose(dq, cos, sin)
        dk = apply_rope_transpose(dk, cos, sin)
    dqkv = np.concatenate([dq.reshape(B, T, Hq * dh), dk.reshape(B, T, Hkv * dh),
                           dv.reshape(B, T, Hkv * dh)], axis=2)
    grad_w_hat = dqkv.reshape(B * T, -1).T @ x.reshape(B * T, d)
    r = lsq_factor(v, bits)
    if kappa is None or kappa <= 0:
        kappa = default_kappa(bits, G)
    D = grad_w_hat.shape[0]
    grad_s = kappa * (grad_w_hat * r).reshape(D, d // G, G).sum(axis=2)
    return dict(loss=mse + lam_kl * kl, mse=mse, kl=kl, grad_s=grad_s, grad_w_hat=grad_w_hat,
                codes=codes, w_hat=w_hat, a_ref=a_ref, lse_ref=teacher["lse"])


# --------------------------------------------------------------------------------------------
# 7. Sensitivity (Section 2.4, Eq. 5-6; reading R19): forward-mode products and Hutchinson
# --------------------------------------------------------------------------------------------

def attention_jvp(q, k, v, P, dq, dk, dv, scale: float):
    """Jacobian-vector product of causal GQA attention (forward mode): with S = Q K^T * scale,
    dS = (dQ K^T + Q dK^T) * scale on the visible keys, dP = P * (dS - rowsum(P * dS)) (softmax),
    dO = dP V + P dV. Inputs as for attention_vjp, tangents dq [B,T,Hq,d_h], dk/dv [B,T,Hkv,d_h]."""
    B, T, Hq, dh = q.shape
    Hkv = k.shape[2]
    mask = np.triu(np.ones((T, T), dtype=bool), k=1)
    dO = np.empty_like(q)
    for b in range(B):
        for h in range(Hq):
            g = _kv_head(h, Hq, Hkv)
            Ph = P[b, h]
            dS = (dq[b, :, h, :] @ k[b, :, g, :].T + q[b, :, h, :] @ dk[b, :, g, :].T) * scale
            dS = np.where(mask, 0.0, dS)
            dP = Ph * (dS - (Ph * dS).sum(axis=1, keepdims=True))
            dO[b, :, h, :] = dP @ v[b, :, g, :] + Ph @ dv[b, :, g, :]
    return dO


def block_jvp(x: np.ndarray, w: np.ndarray, V: np.ndarray, desc: dict) -> np.ndarray:
    """J_A V: the derivative of A(X; w) [B, T, Hq*d_h] along the weight direction V (shaped like w):
    projection X V^T, the same RoPE rotation (linear), then the attention JVP."""
    B, T, _ = x.shape
    Hq, Hkv, dh = desc["n_q_heads"], desc["n_kv_heads"], desc["head_dim"]
    _, parts = block_forward(x, w, desc, return_parts=True)
    dq, dk, dv = split_heads(project(x, V), Hq, Hkv, dh)
    if desc.get("use_rope", False):
        cos, sin = rope_tables(T, dh, float(desc.get("rope_theta", 10000.0)))
        dq = apply_rope(dq, cos, sin)
        dk = apply_rope(dk, cos, sin)
    dO = attention_jvp(parts["q"], parts["k"], parts["v"], parts["P"], dq, dk, dv,
                       _softmax_scale(desc))
    return dO.reshape(B, T, Hq * dh)


def gn_quadratic_form(x, w, V, desc) -> float:
    """v^T H v at the float point (Eq. 5, lambda_KL = 0): 2 ||J_A v||^2 / n (reading R19)."""
    jv = block_jvp(x, w, V, desc)
    return 2.0 * float((jv ** 2).sum()) / jv.size


_SM64_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_SM64_M1 = np.uint64(0xBF58476D1CE4E5B9)
_SM64_M2 = np.uint64(0x94D049BB133111EB)


def splitmix64(seed: int, counters) -> np.ndarray:
    """Outputs number n + 1 (n = counters) of the SplitMix64 generator seeded with `seed` (Steele,
    Lea and Flood, "Fast splittable pseudorandom number generators", 2014): the state after n + 1
    steps is seed + (n + 1) * gamma (mod 2^64), passed through the generator's mixing function."""
    n = np.asarray(counters, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = np.uint64(seed) + (n + np.uint64(1)) * _SM64_GAMMA
        z = (z ^ (z >> np.uint64(30))) * _SM64_M1
        z = (z ^ (z >> np.uint64(27))) * _SM64_M2
        return z ^ (z >> np.uint64(31))


def rademacher_probe(seed: int, probe: int, shape) -> np.ndarray:
    """Rademacher probe number `probe` (entries +-1) of the Hutchinson estimate: entry e (row-major)
    takes output probe * size + e + 1 of splitmix64(seed); -1 when its top bit is set, else +1."""
    size = int(np.prod(shape))
    z = splitmix64(seed, np.arange(size, dtype=np.uint64) + np.uint64(probe * size))
    return np.where((z >> np.uint64(63)) == 1, -1.0, 1.0).reshape(shape)


def hutchinson_trace(x, w, desc, probes) -> float:
    """Tr(H) ~ (1/m) sum_i v_i^T H v_i over the given Rademacher probes [m, *w.shape] (Hutchinson
    estimator, Section 2.4)."""
    return float(np.mean([gn_quadratic_form(x, w, v, desc) for v in probes]))


def omega_scores(trace: float, w: np.ndarray, s: np.ndarray, bits: int, group_size: int,
                 layers_after: int = 0):
    """Eq. 6: C1 Omega(b) = Tr(H) ||Q_b(W) - W||_F^2 and C2 = (L - i) Omega(b), with
    layers_after = L - i. Returns (c1, c2)."""
    _, w_hat, _ = quantize(w, s, bits, group_size)
    c1 = trace * float(((w_hat - w) ** 2).sum())
    return c1, layers_after * c1


# --------------------------------------------------------------------------------------------
# 8. Allocation (Section 2.4, Eq. 7; App. B "Allocators"; reading R20)
# --------------------------------------------------------------------------------------------

def pareto_frontier(costs, omegas):
    """Indices of the non-dominated points of one layer, given in increasing cost: point k is kept
    when every cheaper point has a strictly larger Omega."""
    keep, best = [], None
    for k, om in enumerate(omegas):
        if best is None or om < best:
            keep.append(k)
            best = om
    return keep


def allocate_bits(omega, widths, n_weights, avg_bits: float, method: str = "greedy"):
    """min sum_i Omega_i(b_i) s.t. sum_i n_i b_i <= avg_bits * sum_i n_i (Eq. 7), by the greedy walk
    (method "greedy") or the same walk on each layer's Pareto frontier ("pareto"). omega [L, K] for
    the increasing widths [K]. Returns the chosen width of every layer."""
    omega = [[float(v) for v in row] for row in omega]
    widths = [int(b) for b in widths]
    n = [int(v) for v in n_weights]
    L = len(omega)
    budget = float(avg_bits) * float(sum(n))
    if method == "greedy":
        cand = [list(range(len(widths))) for _ in range(L)]
    elif method == "pareto":
        cand = [pareto_frontier([n[i] * b for b in widths], omega[i]) for i in range(L)]
    else:
        raise ValueError(method)
    if sum(n[i] * widths[cand[i][0]] for i in range(L)) > budget:
        raise ValueError("budget below the cheapest allocation")
    pos = [len(c) - 1 for c in cand]                       # start at the highest width
    cost = sum(n[i] * widths[cand[i][pos[i]]] for i in range(L))

    def width(i, p):
        return widths[cand[i][p]]

    def om(i, p):
        return omega[i][cand[i][p]]

    while cost > budget:                                   # downgrades: least damage per bit saved
        best, pick = None, None
        for i in range(L):
            if pos[i] == 0:
                continue
            dc = n[i] * (width(i, pos[i]) - width(i, pos[i] - 1))
            r = (om(i, pos[i] - 1) - om(i, pos[i])) / dc
            if best is None or r < best:
                best, pick = r, i
        cost -= n[pick] * (width(pick, pos[pick]) - width(pick, pos[pick] - 1))
        pos[pick] -= 1
    while True:                                            # leftovers: best gain per bit that fits
        best, pick = None, None
        for i in range(L):
            if pos[i] + 1 == len(cand[i]):
                continue
            dc = n[i] * (width(i, pos[i] + 1) - width(i, pos[i]))
            gain = om(i, pos[i]) - om(i, pos[i] + 1)
            if cost + dc > budget or not gain > 0:
                continue
            r = gain / dc
            if best is None or r > best:
                best, pick = r, i
        if pick is None:
            break
        cost += n[pick] * (width(pick, pos[pick] + 1) - width(pick, pos[pick]))
        pos[pick] += 1
    return [width(i, pos[i]) for i in range(L)]

