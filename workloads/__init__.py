"""Seeded synthetic inputs for the joint attention-block loss (JAB) workloads.

This module only draws random tensors with the shapes and value distributions of the
GPT-2-small and Mistral-7B attention blocks the paper studies (Section 3 and App. C,
"Models and scope"). It holds none of the method's arithmetic: no quantizer, no
projection, no attention. Both the float64 oracle (through the tests) and the CUDA path
receive the same bf16 bytes from here.

The paper's activations come from WikiText-2 / C4 calibration text fed through the real
models; neither the models nor the corpora are available, so these seeded synthetic
inputs stand in for them:

* X ~ N(0, 1), or Student-t(df) rescaled to unit variance (divide by sqrt(df/(df-2))),
  built exactly from normals as Z / sqrt(chi2_df / df);
* "outlier channels": a seeded subset of ceil(p * d_model) input channels multiplied by
  a constant factor, mimicking the heavy activation channels of LLMs;
* weights W_q, W_k, W_v ~ N(0, sigma^2), rounded to bf16 once, in nn.Linear layout
  (rows = output features, Q rows then K rows then V rows).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional, Tuple

import torch

__all__ = ["BlockShape", "Workload", "WORKLOADS", "make_x", "make_w", "make_block_weights"]


@dataclass(frozen=True)
class BlockShape:
    """Shape of one attention block (Section 2.1: d, n_head, d_head; GQA and RoPE for Mistral)."""

    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    use_rope: bool
    rope_theta: float = 10000.0

    @property
    def d_out(self) -> int:
        """Rows of the joint weight [W_Q | W_K | W_V] in nn.Linear layout."""
        return (self.n_q_heads + 2 * self.n_kv_heads) * self.head_dim


GPT2_SMALL = BlockShape(d_model=768, n_q_heads=12, n_kv_heads=12, head_dim=64, use_rope=False)
MISTRAL_7B = BlockShape(d_model=4096, n_q_heads=32, n_kv_heads=8, head_dim=128, use_rope=True,
                        rope_theta=10000.0)


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: block shape, calibration batch, candidate bit widths."""

    name: str
    shape: BlockShape
    batch: int
    seq_len: int
    group_size: int
    bits: Tuple[int, ...]
    x_dist: str                      # "normal" or "student_t"
    x_df: Optional[int] = None       # degrees of freedom for student_t
    outlier_frac: float = 0.0
    outlier_factor: float = 1.0
    w_std: float = 0.02
    n_blocks: int = 1                # independent seeded blocks (sensitivity table)
    scale_init: str = "absmax"       # "absmax" or "minmse"
    mode: str = "fwd"                # "fwd" (loss per candidate) or "fwd_bwd"
    seed: int = 0

    @property
    def tokens(self) -> int:
        return self.batch * self.seq_len

    def with_batch(self, batch: int, seq_len: Optional[int] = None) -> "Workload":
        """Same distribution and block, fewer sequences (for bounded oracle samples)."""
        from dataclasses import replace
        return replace(self, batch=batch, seq_len=self.seq_len if seq_len is None else seq_len)


WORKLOADS = {
    # GPT-2-small block, oracle smoke test: X fp32 N(0,1) rounded to bf16 once.
    "gpt2_smoke": Workload("gpt2_smoke", GPT2_SMALL, batch=4, seq_len=128, group_size=128,
                           bits=(3,), x_dist="normal", w_std=0.02, mode="fwd_bwd", seed=0),
    # GPT-2-small sensitivity sweep: 1% outlier channels x20, candidates {2,3,4,8}.
    "gpt2_sweep": Workload("gpt2_sweep", GPT2_SMALL, batch=64, seq_len=1024, group_size=128,
                           bits=(2, 3, 4, 8), x_dist="normal", outlier_frac=0.01,
                           outlier_factor=20.0, w_std=0.02, mode="fwd", seed=0),
    # Mistral-7B block: Student-t(4) unit variance, 3-bit, fwd + STE backward.
    "mistral_block": Workload("mistral_block", MISTRAL_7B, batch=128, seq_len=2048, group_size=128,
                              bits=(3,), x_dist="student_t", x_df=4, w_std=0.015,
                              mode="fwd_bwd", seed=0),
    # Mistral-7B sensitivity table: 32 blocks x {2,3,4,5,8}, 0.5% outlier channels x30.
    "mistral_scoring": Workload("mistral_scoring", MISTRAL_7B, batch=32, seq_len=2048,
                                group_size=128, bits=(2, 3, 4, 5, 8), x_dist="student_t", x_df=4,
                                outlier_frac=0.005, outlier_factor=30.0, w_std=0.015,
                                n_blocks=32, mode="fwd", seed=0),
    # Mistral-7B STE fitting step at long context: Student-t(3), 1% outliers x20, 2-bit G=64,
    # min-MSE warm-start scales.
    "mistral_ste_long": Workload("mistral_ste_long", MISTRAL_7B, batch=16, seq_len=4096,
                                 group_size=64, bits=(2,), x_dist="student_t", x_df=3,
                                 outlier_frac=0.01, outlier_factor=20.0, w_std=0.015,
                                 scale_init="minmse", mode="fwd_bwd", seed=0),
}


def _generator(device, seed: int) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def make_x(wl: Workload, device="cpu", seed: Optional[int] = None, batch: Optional[int] = None,
           seq_len: Optional[int] = None) -> torch.Tensor:
    """Calibration activations X [B, T, d_model] as bf16, seeded.

    The outlier channel subset is drawn first from the same generator, so it does not
    depend on B or T. Sequences are drawn one after another, so the first k sequences of
    a batch are the same tensor for any B >= k.
    """
    seed = wl.seed if seed is None else seed
    B = wl.batch if batch is None else batch
    T = wl.seq_len if seq_len is None else seq_len
    d = wl.shape.d_model
    g = _generator(device, seed)
    n_out = int(math.ceil(wl.outlier_frac * d)) if wl.outlier_frac > 0 else 0
    perm = torch.randperm(d, generator=g, device=device)
    outlier_idx = perm[:n_out]
    x = torch.empty((B, T, d), dtype=torch.bfloat16, device=device)
    for b in range(B):
        if wl.x_dist == "normal":
            xb = torch.randn((T, d), generator=g, device=device, dtype=torch.float32)
        elif wl.x_dist == "student_t":
            df = int(wl.x_df)
            z = torch.randn((T, d), generator=g, device=device, dtype=torch.float32)
            chi2 = torch.zeros((T, d), device=device, dtype=torch.float32)
            for _ in range(df):
                chi2 += torch.randn((T, d), generator=g, device=device, dtype=torch.float32) ** 2
            xb = z / torch.sqrt(chi2 / df)
            xb = xb / math.sqrt(df / (df - 2.0))
        else:
            raise ValueError(f"unknown x_dist {wl.x_dist!r}")
        if n_out:
            xb[:, outlier_idx] *= wl.outlier_factor
        x[b] = xb.to(torch.bfloat16)
    return x


def make_w(shape: BlockShape, w_std: float, device="cpu", seed: int = 0) -> torch.Tensor:
    """Joint weight [W_Q; W_K; W_V] as bf16 [(Hq + 2 Hkv) * d_h, d_model], N(0, w_std^2)."""
    g = _generator(device, seed + 7919)
    w = torch.randn((shape.d_out, shape.d_model), generator=g, device=device, dtype=torch.float32)
    return (w * w_std).to(torch.bfloat16)


def make_block_weights(wl: Workload, block: int = 0, device="cpu") -> torch.Tensor:
    """Weights of block `block`; block i of a multi-block workload is seeded with seed + 1 + i."""
    seed = wl.seed if wl.n_blocks == 1 else wl.seed + 1 + block
    return make_w(wl.shape, wl.w_std, device=device, seed=seed)
