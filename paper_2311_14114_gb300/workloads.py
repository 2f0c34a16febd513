"""Seeded synthetic workloads for SONIQ's inference hot path.

This module only draws inputs: activations, weights, the per-channel
precision assignment and the channel permutation that SONIQ-QAT would hand to
inference (Sec. 3 "Dynamic channel re-ordering"; Alg. 1 Phase I).  It holds
none of the method's arithmetic (no scales, codes, packing or products), so
both the CUDA path and the CPU oracle may consume what it returns.

The paper evaluates on IWSLT14, CIFAR-10/100 and ImageNet models (Sec. 5);
none of those datasets or trained weights exist here.  These generators stand
in for their layer shapes with Gaussian data:

  * activations ~ N(0, 1) in fp16 (conv inputs pass through ReLU), with a few
    seeded outlier channels scaled up; outlier channels are always assigned
    the high precision (Sec. 1: harder channels get more bits);
  * weights ~ N(0, std) in fp32;
  * the high-precision channel count is floor(frac * K + 0.5); the remaining
    high channels are a seeded choice among the non-outliers;
  * the permutation lists low channels then high channels, each ascending.

Random draws, in order, from ``numpy.random.default_rng(seed)``: outlier
channels, extra high channels, activations, weights.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Tuple

import numpy as np


@dataclasses.dataclass(frozen=True)
class LinearSpec:
    name: str
    M: int
    K: int
    N: int
    bits_lo: int
    bits_hi: int
    frac_hi: float
    n_outliers: int = 0
    outlier_scale: float = 1.0
    w_std: float = 0.02
    seed: int = 0

    @property
    def ops(self) -> int:
        """Algorithmic integer ops: 2*M*N*K with the logical (unpadded) K."""
        return 2 * self.M * self.N * self.K


@dataclasses.dataclass(frozen=True)
class ConvSpec:
    name: str
    batch: int
    H: int
    W: int
    C: int
    C_out: int
    R: int
    S: int
    stride: Tuple[int, int]
    pad: Tuple[int, int]
    bits_lo: int
    bits_hi: int
    frac_hi: float
    relu: bool = True
    w_std: Optional[float] = None   # default sqrt(2 / (R*S*C))
    seed: int = 0

    @property
    def out_hw(self) -> Tuple[int, int]:
        P = (self.H + 2 * self.pad[0] - self.R) // self.stride[0] + 1
        Q = (self.W + 2 * self.pad[1] - self.S) // self.stride[1] + 1
        return P, Q

    @property
    def M(self) -> int:
        P, Q = self.out_hw
        return self.batch * P * Q

    @property
    def K(self) -> int:
        return self.R * self.S * self.C

    @property
    def ops(self) -> int:
        return 2 * self.M * self.C_out * self.K


def high_count(K: int, frac: float) -> int:
    return int(np.floor(frac * K + 0.5))


def assignment(rng: np.random.Generator, K: int, frac_hi: float, n_outliers: int):
    """Per-channel precision assignment and the inference permutation.

    Returns (perm, count, outliers): perm[j] is the original channel at packed
    position j (low group first, both groups ascending), count = [low, high]."""
    c_hi = high_count(K, frac_hi)
    n_out = min(n_outliers, c_hi)
    outliers = np.sort(rng.choice(K, size=n_out, replace=False)) if n_out else np.zeros(0, np.int64)
    others = np.setdiff1d(np.arange(K), outliers)
    extra = rng.choice(others, size=c_hi - n_out, replace=False) if c_hi > n_out else np.zeros(0, np.int64)
    high = np.zeros(K, dtype=bool)
    high[outliers] = True
    high[extra] = True
    perm = np.concatenate([np.flatnonzero(~high), np.flatnonzero(high)]).astype(np.int32)
    return perm, [int(K - c_hi), int(c_hi)], outliers


def make_linear(spec: LinearSpec, M: Optional[int] = None) -> Dict[str, object]:
    """A fp16 [M][K], W fp32 [N][K], perm, count, bits."""
    M = spec.M if M is None else M
    rng = np.random.default_rng(spec.seed)
    perm, count, outliers = assignment(rng, spec.K, spec.frac_hi, spec.n_outliers)
    A = rng.standard_normal((M, spec.K), dtype=np.float32)
    if len(outliers):
        A[:, outliers] *= spec.outlier_scale
    W = rng.standard_normal((spec.N, spec.K), dtype=np.float32) * np.float32(spec.w_std)
    return dict(A=A.astype(np.float16), W=W.astype(np.float32), perm=perm, count=count,
                bits=[spec.bits_lo, spec.bits_hi], outliers=outliers)


def make_conv(spec: ConvSpec) -> Dict[str, object]:
    """X fp16 NHWC [batch][H][W][C], W fp32 OHWI [C_out][R*S][C], perm, count, bits."""
    rng = np.random.default_rng(spec.seed)
    perm, count, outliers = assignment(rng, spec.C, spec.frac_hi, 0)
    X = rng.standard_normal((spec.batch, spec.H, spec.W, spec.C), dtype=np.float32)
    if spec.relu:
        X = np.maximum(X, 0.0)
    std = spec.w_std if spec.w_std is not None else float(np.sqrt(2.0 / (spec.R * spec.S * spec.C)))
    Wt = rng.standard_normal((spec.C_out, spec.R * spec.S, spec.C), dtype=np.float32) * np.float32(std)
    return dict(X=X.astype(np.float16), W=Wt.astype(np.float32), perm=perm, count=count,
                bits=[spec.bits_lo, spec.bits_hi])


# ---------------------------------------------------------------------------
# The five workload families (layer shapes of the paper's benchmarks).
# ---------------------------------------------------------------------------

LINEAR_SMALL = LinearSpec("linear_64x512x512_2b8b", M=64, K=512, N=512, bits_lo=2, bits_hi=8,
                          frac_hi=0.25, n_outliers=4, outlier_scale=10.0)

CONV_RESNET = ConvSpec("conv_resnet18_64x14x14x256_3x3_4b8b", batch=64, H=14, W=14, C=256,
                       C_out=256, R=3, S=3, stride=(1, 1), pad=(1, 1), bits_lo=4, bits_hi=8,
                       frac_hi=0.30)
CONV_RESNET_1B4B = dataclasses.replace(CONV_RESNET, name="conv_resnet18_64x14x14x256_3x3_1b4b",
                                       bits_lo=1, bits_hi=4)

MLP_UP = LinearSpec("mlp_up_16384x768x3072_2b8b", M=16384, K=768, N=3072, bits_lo=2, bits_hi=8,
                    frac_hi=0.20, n_outliers=8, outlier_scale=20.0)

DECODE = {m: LinearSpec(f"decode_m{m}_4096x11008_3b6b", M=m, K=4096, N=11008, bits_lo=3,
                        bits_hi=6, frac_hi=0.15)
          for m in (1, 4, 16)}


def sweep_specs() -> List[LinearSpec]:
    out = []
    for lo in (1, 2, 3, 4):
        for hi in (4, 6, 8):
            for frac in (0.0, 0.10, 0.25, 0.50, 1.00):
                out.append(LinearSpec(f"sweep_8192x4096x4096_lo{lo}_hi{hi}_f{int(frac * 100)}",
                                      M=8192, K=4096, N=4096, bits_lo=lo, bits_hi=hi,
                                      frac_hi=frac))
    return out


# The precision-sweep point the benchmark headline is quoted on: 4-bit low,
# 8-bit high, 25 % of the 4096 channels (1024) at 8 bits.
SWEEP_HEADLINE = LinearSpec("sweep_8192x4096x4096_lo4_hi8_f25", M=8192, K=4096, N=4096, bits_lo=4,
                            bits_hi=8, frac_hi=0.25)


def random_linear(seed: int, M: int, K: int, N: int, bits_lo: int, bits_hi: int,
                  frac_hi: float, n_outliers: int = 0, outlier_scale: float = 8.0):
    """Small seeded case for parity sweeps."""
    return make_linear(LinearSpec(f"rand_{seed}", M=M, K=K, N=N, bits_lo=bits_lo,
                                  bits_hi=bits_hi, frac_hi=frac_hi, n_outliers=n_outliers,
                                  outlier_scale=outlier_scale, seed=seed))


# ---------------------------------------------------------------------------
# Phase II workload (Algorithm 1, Phase II: quantized fine-tuning): a
# transformer MLP block (up, then down projection) whose fp32 master weights
# are quantized on the fly in every step; precisions per channel as Phase I
# would leave them (about 15 % of the channels at the higher width).
# ---------------------------------------------------------------------------

@dataclasses.dataclass(frozen=True)
class Phase2Spec:
    name: str
    M: int                      # tokens per step
    widths: Tuple[int, ...]     # layer widths: input, hidden..., output
    bits: Tuple[int, int]       # (low, high) bits of every layer
    frac_hi: float
    seed: int = 0
    w_std: float = 0.02
    sub_k: int = 0              # scale runs along K (0: one scale per group)


PHASE2_MLP = Phase2Spec("phase2_mlp_2048x4096x11008x4096_3b6b", M=2048, widths=(4096, 11008, 4096),
                        bits=(3, 6), frac_hi=0.15)


def make_phase2(spec: Phase2Spec, M: Optional[int] = None) -> Dict[str, object]:
    """Input X fp16 [M][widths[0]] and, per layer, fp32 master weights with
    their channel permutation and group sizes."""
    M = spec.M if M is None else M
    rng = np.random.default_rng(spec.seed)
    X = rng.standard_normal((M, spec.widths[0]), dtype=np.float32).astype(np.float16)
    layers = []
    for K, N in zip(spec.widths[:-1], spec.widths[1:]):
        perm, count, _ = assignment(rng, K, spec.frac_hi, 0)
        W = rng.standard_normal((N, K), dtype=np.float32) * np.float32(spec.w_std)
        layers.append(dict(W=W, perm=perm, count=count, bits=list(spec.bits)))
    return dict(X=X, layers=layers)
