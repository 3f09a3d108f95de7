"""Seeded synthetic inputs for the RFQ linear layer.

This module holds input generation only -- none of the method's arithmetic --
so both the CUDA path and the CPU oracle consume the exact same bytes.

The paper's activations (Qwen3-VL and Wan2.2 linear layers, Sec. 5) and its
datasets are not available, so the activations are drawn from seeded
distributions shaped like the paper's description of them (Sec. 4.2: heavy
tails, outlier channels, massive-activation tokens):

  body          N(0,1), Student-t(nu=3) or Laplace(0, b), drawn in float64
                from numpy's Philox bit generator seeded with ``seed``
  outlier chans round(frac * K) distinct columns, chosen by a seeded
                permutation, multiplied by ``chan_scale``
  outlier toks  round(frac * M) distinct rows, chosen likewise, multiplied
                by ``tok_scale``
  rounding      float32 -> bf16 with round-to-nearest-even on the bit pattern

Weights are N(0, 0.02) in bf16, laid out [K, N] row-major.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


def f32_to_bf16_bits(f: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round-to-nearest-even); returns uint16."""
    u = np.ascontiguousarray(f, np.float32).view(np.uint32)
    lsb = (u >> 16) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass(frozen=True)
class ActSpec:
    """Distribution of a synthetic activation matrix X [M, K]."""
    M: int
    K: int
    body: str = "normal"          # normal | student_t3 | laplace
    body_scale: float = 1.0       # sigma (normal) or b (laplace)
    chan_frac: float = 0.0        # fraction of outlier channels (columns)
    chan_count: int | None = None  # explicit count, overrides chan_frac
    chan_scale: float = 1.0
    tok_frac: float = 0.0         # fraction of massive-activation tokens (rows)
    tok_count: int | None = None
    tok_scale: float = 1.0
    seed: int = 0


@dataclass(frozen=True)
class LinearSpec:
    name: str
    act: ActSpec
    N: int = 0                    # 0: activation-only workload
    w_std: float = 0.02
    fmt: str = "mxfp4"            # mxfp4 | hif4
    notes: dict = field(default_factory=dict)
    groups: int = 0               # > 0: act.M token rows routed over this many experts (grouped GEMM)


def make_group_counts(rows: int, groups: int, seed: int = 0) -> np.ndarray:
    """Rows per group for a routed (mixture-of-experts) workload: a
    multinomial draw of `rows` over `groups` with seeded, unevenly spread
    probabilities (softmax of standard normal logits)."""
    rng = np.random.default_rng(seed + 7919)
    logits = rng.standard_normal(groups)
    p = np.exp(logits - logits.max())
    return rng.multinomial(rows, p / p.sum())


def group_layout(counts: np.ndarray, align: int = 128):
    """Row layout of routed groups: every group starts on a multiple of
    `align` rows.  Returns (starts [G], ends [G], padded total rows)."""
    starts, pos = [], 0
    for c in counts:
        starts.append(pos)
        pos = -(-(pos + int(c)) // align) * align
    starts = np.array(starts, np.int64)
    return starts, starts + np.asarray(counts, np.int64), max(pos, align)


def _count(frac, count, dim):
    if count is not None:
        return int(count)
    return int(round(frac * dim))


def make_activation(spec: ActSpec) -> np.ndarray:
    """bf16 bit patterns (uint16) of shape [M, K]."""
    rng = np.random.Generator(np.random.Philox(spec.seed))
    M, K = spec.M, spec.K
    if spec.body == "normal":
        x = rng.standard_normal((M, K), dtype=np.float32)
        if spec.body_scale != 1.0:
            x *= np.float32(spec.body_scale)
    elif spec.body == "student_t3":
        x = rng.standard_t(3.0, size=(M, K)).astype(np.float32)
    elif spec.body == "laplace":
        x = rng.laplace(0.0, spec.body_scale, size=(M, K)).astype(np.float32)
    else:
        raise ValueError(f"unknown body {spec.body!r}")
    nc = _count(spec.chan_frac, spec.chan_count, K)
    if nc:
        cols = np.sort(rng.permutation(K)[:nc])
        x[:, cols] *= np.float32(spec.chan_scale)
    nt = _count(spec.tok_frac, spec.tok_count, M)
    if nt:
        rows = np.sort(rng.permutation(M)[:nt])
        x[rows, :] *= np.float32(spec.tok_scale)
    return f32_to_bf16_bits(x)


def make_weight(K: int, N: int, std: float = 0.02, seed: int = 0) -> np.ndarray:
    """bf16 bit patterns (uint16) of W [K, N] ~ N(0, std^2)."""
    rng = np.random.Generator(np.random.Philox(seed + 0x5EED))
    w = rng.standard_normal((K, N), dtype=np.float32) * np.float32(std)
    return f32_to_bf16_bits(w)


# The workloads: shapes of the paper's model families (Qwen3-VL-8B and -30B-A3B
# projections and a Wan2.2-14B DiT FFN), with seeded synthetic values.
WORKLOADS = {
    "tiny": LinearSpec(
        "tiny_rfq_linear_128x512x512",
        ActSpec(128, 512, "normal", chan_count=4, chan_scale=64.0, seed=0),
        N=512),
    "act_quant": LinearSpec(
        "act_quant_16384x4096_student_t3",
        ActSpec(16384, 4096, "student_t3", chan_frac=0.005, chan_scale=100.0, seed=1)),
    "qwen_gate_up": LinearSpec(
        "qwen3vl8b_gate_up_4096x4096x24576",
        ActSpec(4096, 4096, "normal", chan_frac=0.01, chan_scale=50.0,
                tok_count=8, tok_scale=500.0, seed=2),
        N=24576),
    "qwen_down_hif4": LinearSpec(
        "qwen3vl8b_down_hif4_4096x12288x4096",
        ActSpec(4096, 12288, "laplace", body_scale=0.3, chan_frac=0.01, chan_scale=50.0, seed=3),
        N=4096, fmt="hif4"),
    # Qwen3-VL-30B-A3B expert gate/up projection (hidden 2048, 2 x 768 expert
    # width, 128 experts, 8 per token): 4096 tokens give 32768 routed rows.
    "qwen_moe_gate_up": LinearSpec(
        "qwen3vl30b_a3b_moe_gate_up_32768x2048x1536_128experts",
        ActSpec(32768, 2048, "normal", chan_frac=0.01, chan_scale=50.0, tok_count=8, tok_scale=500.0, seed=5),
        N=1536, groups=128),
    "wan_ffn_up": LinearSpec(
        "wan22_14b_ffn_up_32760x5120x13824",
        ActSpec(32760, 5120, "normal", chan_frac=0.01, chan_scale=64.0,
                tok_frac=0.001, tok_scale=200.0, seed=4),
        N=13824),
}
