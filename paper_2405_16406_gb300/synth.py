"""Seeded synthetic inputs with the shapes and value distributions of the
LLaMA-style layers the rotated W4A4 path runs on.

This module holds no arithmetic of the method (no rotation, no quantizer,
no GEMM): it only draws random fp16 tensors.  Both the CUDA path and the CPU
oracle consume exactly the bytes produced here.

Recipe (one ``numpy.random.default_rng(seed)`` per workload, drawn in fp32,
rounded once to fp16):

* activations ~ N(0, 1), with a seeded set of distinct "outlier" columns,
  shared by all tokens, multiplied by a fixed factor;
* SwiGLU-like activations (down_proj input) = a * SiLU(b), a, b ~ N(0, 1);
* weights ~ N(0, 0.02);
* Q/K/V ~ N(0, 1) with a few fixed head_dim channels (same for every head,
  token and tensor) multiplied by a factor.

They stand in for real LLaMA-2/3 activations and weights and for the
WikiText2 / zero-shot data the paper evaluates on, none of which is used.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Dict, Optional, Tuple

import numpy as np


def _outlier_cols(rng: np.random.Generator, K: int, count: int) -> np.ndarray:
    return np.sort(rng.choice(K, size=count, replace=False))


def activations(rng: np.random.Generator, M: int, K: int, outlier_frac: Optional[float] = None,
                outlier_count: Optional[int] = None, factor: float = 1.0,
                swiglu: bool = False) -> np.ndarray:
    """fp16 [M, K]: N(0,1) (or a*SiLU(b)) with outlier columns scaled."""
    if swiglu:
        a = rng.standard_normal((M, K), dtype=np.float32)
        b = rng.standard_normal((M, K), dtype=np.float32)
        x = a * (b / (1.0 + np.exp(-b)))
    else:
        x = rng.standard_normal((M, K), dtype=np.float32)
    n_out = outlier_count if outlier_count is not None else int(round((outlier_frac or 0.0) * K))
    if n_out > 0:
        cols = _outlier_cols(rng, K, n_out)
        x[:, cols] *= np.float32(factor)
    return x.astype(np.float16)


def weights(rng: np.random.Generator, N: int, K: int, std: float = 0.02) -> np.ndarray:
    return (rng.standard_normal((N, K), dtype=np.float32) * np.float32(std)).astype(np.float16)


@dataclass
class LinearCase:
    name: str
    M: int
    K: int
    N: int
    had: Optional[Tuple[int, int]]   # (n_small, n_pow2) or None
    act_symmetric: bool
    clip: float
    x: np.ndarray = field(repr=False)
    w: np.ndarray = field(repr=False)


@dataclass
class KVCase:
    name: str
    B: int
    S: int
    Hq: int
    Hkv: int
    D: int
    had: Tuple[int, int]
    clip: float
    q: np.ndarray = field(repr=False)
    k: np.ndarray = field(repr=False)
    v: np.ndarray = field(repr=False)


# ---------------------------------------------------------------------------
# The five workloads (sizes exactly as specified; ``scale`` shrinks M / S for
# oracle-sized parity runs without changing K, N, the rotation or the mix).
# ---------------------------------------------------------------------------
def tiny_linear(seed: int = 0) -> LinearCase:
    """16 tokens x 256 -> 512, Sylvester H256 online, symmetric activations."""
    rng = np.random.default_rng(seed)
    x = activations(rng, 16, 256, outlier_count=4, factor=50.0)
    w = weights(rng, 512, 256)
    return LinearCase("tiny_16x256x512_h256", 16, 256, 512, (1, 256), True, 1.0, x, w)


def llama3_8b_gate_up(seed: int = 0, M: int = 2048) -> LinearCase:
    """LLaMA-3-8B gate/up: M x 4096 -> 14336, no online rotation, asym acts."""
    rng = np.random.default_rng(seed)
    x = activations(rng, M, 4096, outlier_frac=0.01, factor=30.0)
    w = weights(rng, 14336, 4096)
    return LinearCase(f"llama3_8b_gate_up_M{M}", M, 4096, 14336, None, False, 1.0, x, w)


def llama3_8b_down_proj(seed: int = 0, M: int = 2048) -> LinearCase:
    """LLaMA-3-8B down_proj: M x 14336 -> 4096, online R4 = H28 (x) H512,
    SwiGLU-like activations, symmetric activations."""
    rng = np.random.default_rng(seed)
    x = activations(rng, M, 14336, outlier_frac=0.005, factor=100.0, swiglu=True)
    w = weights(rng, 4096, 14336)
    return LinearCase(f"llama3_8b_down_proj_M{M}", M, 14336, 4096, (28, 512), True, 1.0, x, w)


def llama32_3b_up(seed: int = 0, M: int = 8192) -> LinearCase:
    """LLaMA-3.2-3B-like hidden 3072 -> 8192 with online H12 (x) H256."""
    rng = np.random.default_rng(seed)
    x = activations(rng, M, 3072, outlier_frac=0.01, factor=30.0)
    w = weights(rng, 8192, 3072)
    return LinearCase(f"llama32_3b_up_M{M}", M, 3072, 8192, (12, 256), False, 1.0, x, w)


def llama32_3b_down(seed: int = 0, M: int = 8192) -> LinearCase:
    """LLaMA-3.2-3B-like intermediate 8192 -> 3072 with online H8192."""
    rng = np.random.default_rng(seed)
    x = activations(rng, M, 8192, outlier_frac=0.01, factor=30.0)
    w = weights(rng, 3072, 8192)
    return LinearCase(f"llama32_3b_down_M{M}", M, 8192, 3072, (1, 8192), False, 1.0, x, w)


def kv_case(seed: int = 0, B: int = 8, S: int = 4096, Hq: int = 32, Hkv: int = 8,
            D: int = 128) -> KVCase:
    """Q/K/V ~ N(0,1) with 2 fixed head_dim channels x20; Sylvester H_D."""
    rng = np.random.default_rng(seed)
    cols = _outlier_cols(rng, D, 2)

    def draw(H):
        t = rng.standard_normal((B, S, H, D), dtype=np.float32)
        t[..., cols] *= np.float32(20.0)
        return t.astype(np.float16)

    q = draw(Hq)
    k = draw(Hkv)
    v = draw(Hkv)
    return KVCase(f"kv_B{B}_S{S}_Hq{Hq}_Hkv{Hkv}_D{D}", B, S, Hq, Hkv, D, (1, D), 1.0, q, k, v)


LINEAR_BUILDERS: Dict[str, callable] = {
    "tiny": tiny_linear,
    "gate_up": llama3_8b_gate_up,
    "down_proj": llama3_8b_down_proj,
    "l32_up": llama32_3b_up,
    "l32_down": llama32_3b_down,
}
