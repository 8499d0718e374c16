"""Seeded synthetic inputs for the OffQ W4A4 linear path.

This module only draws random numbers and lays them out in the shapes of the
Llama-style layers the method targets. It holds none of the method's arithmetic
(no rotation, offset, quantization or GEMM), so both the CUDA path and the CPU
oracle can consume its output without sharing any computation.

Recipe (stands in for the calibration / evaluation activations of the paper's
experiments, which are not available here):

* Activations are generated in the basis the online path sees, i.e. after the
  offline top-1 PCA rotation has concentrated the dominant outlier direction
  into channel 0 (paper Sec. 3.1, Eq. 3). Channel 0 carries the largest outlier;
  further outlier channels sit at c_k = k * floor(K / n_out). Every token carries
  the outliers, with magnitude ``mult * std * (1 + 0.1 * z_t)``, z_t ~ N(0, 1)
  per token ("jitter"), positive sign.
* Bulk entries are N(0, 1) or Student-t(nu=3) (heavy-tailed), in fp32, then
  optionally cast to bf16 (round to nearest even by torch); both sides consume
  the cast values.
* Weights are N(0, 0.02) in fp32.
* KV vectors are N(0, 1) per (token, head) with a channel-0 outlier.
"""

from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional, Tuple

import numpy as np

# Seeds fixed per role: 0 for activations, 1 for weights, 2 for KV.
SEED_X = 0
SEED_W = 1
SEED_KV = 2


def outlier_channels(K: int, n_out: int) -> List[int]:
    """Fixed outlier channel indices c_k = k * floor(K / n_out), k = 0..n_out-1."""
    if n_out <= 0:
        return []
    step = K // n_out
    return [k * step for k in range(n_out)]


def activations(T: int, K: int, *, seed: int = SEED_X, dist: str = "normal",
                n_out: int = 0, mult: float = 0.0, jitter: float = 0.1,
                std: float = 1.0) -> np.ndarray:
    """Token rows X [T, K] float32 with structured outlier channels.

    ``dist`` is ``"normal"`` (N(0, std^2)) or ``"student_t3"`` (Student-t with
    3 degrees of freedom, unscaled, times ``std``).
    """
    rng = np.random.default_rng(seed)
    if dist == "normal":
        x = rng.standard_normal((T, K), dtype=np.float64) * std
    elif dist == "student_t3":
        x = rng.standard_t(3.0, size=(T, K)) * std
    else:
        raise ValueError(f"unknown distribution {dist!r}")
    if n_out > 0 and mult != 0.0:
        z = rng.standard_normal(T)
        amp = mult * std * (1.0 + jitter * z)
        for c in outlier_channels(K, n_out):
            x[:, c] = amp
    return x.astype(np.float32)


def weights(N: int, K: int, *, seed: int = SEED_W, std: float = 0.02) -> np.ndarray:
    """Linear-layer weights W [N, K] float32, N(0, std^2)."""
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((N, K), dtype=np.float64) * std).astype(np.float32)


def kv_heads(T: int, H: int, hd: int, *, seed: int = SEED_KV,
             mult: float = 20.0) -> np.ndarray:
    """Post-RoPE K (or V) vectors [T, H, hd] float32 with a channel-0 outlier per head."""
    rng = np.random.default_rng(seed)
    x = rng.standard_normal((T, H, hd), dtype=np.float64)
    if mult != 0.0:
        z = rng.standard_normal((T, H))
        x[:, :, 0] = mult * (1.0 + 0.1 * z)
    return x.astype(np.float32)


def to_bf16(x: np.ndarray):
    """Round an fp32 array to bf16 (torch RNE cast). Returns a torch CPU tensor."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16)


def bf16_to_f64(t) -> np.ndarray:
    """Exact widening of a torch bf16 tensor to a float64 numpy array."""
    import torch
    return t.to(torch.float64).numpy()


def unit_index_sample(n: int, k: int, *, seed: int = 7) -> np.ndarray:
    """A sorted, seeded sample of k distinct indices out of n (all if k >= n)."""
    if k >= n:
        return np.arange(n)
    rng = np.random.default_rng(seed)
    return np.sort(rng.choice(n, size=k, replace=False))


# --------------------------------------------------------------------------
# Workload table: the Llama-shaped layers the path is measured on.
# Block size g of the online Hadamard / offset per input dim K: the largest
# power of two that is a K-block as listed (K itself when K is a power of two).
# --------------------------------------------------------------------------

BLOCK_FOR_K: Dict[int, int] = {
    512: 512,
    4096: 4096,
    8192: 8192,
    11008: 256,     # 43 blocks
    14336: 1024,    # 14 blocks
    28672: 1024,    # 28 blocks
    128: 128,       # KV head dim
}


def block_for(K: int) -> int:
    if K in BLOCK_FOR_K:
        return BLOCK_FOR_K[K]
    g = 1
    while K % (g * 2) == 0 and g * 2 <= 8192:
        g *= 2
    return g


@dataclasses.dataclass(frozen=True)
class Linear:
    """One linear layer y = W x with W [N, K]; ``rotate`` marks an online-Hadamard site."""
    name: str
    K: int
    N: int
    rotate: bool


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    T: int
    layers: Tuple[Linear, ...]
    x_dtype: str                 # "f32" or "bf16"
    dist: str
    n_out: int
    mult: float
    kv_heads: int = 0            # KV4 heads quantized per token (0: none)
    head_dim: int = 128
    description: str = ""


def _llama_layers(hidden: int, inter: int, kv_dim: int) -> Tuple[Linear, ...]:
    # q/k/v/gate/up inputs arrive already in the offset basis (their rotation
    # is fused into the weights offline), as does the o-proj input (per-head
    # rotation fused into W_V / W_O); the down-proj input takes the online
    # group-wise Hadamard H4.
    return (
        Linear("q", hidden, hidden, False),
        Linear("k", hidden, kv_dim, False),
        Linear("v", hidden, kv_dim, False),
        Linear("o", hidden, hidden, False),
        Linear("gate", hidden, inter, False),
        Linear("up", hidden, inter, False),
        Linear("down", inter, hidden, True),
    )


WORKLOADS: Dict[str, Workload] = {
    "toy": Workload(
        name="toy", T=16, layers=(Linear("toy", 512, 512, True),), x_dtype="f32",
        dist="normal", n_out=2, mult=50.0,
        description="toy OffQ linear: X fp32 [16 x 512] N(0,1) + 2 outlier channels x50 "
                    "with per-token jitter; W fp32 [512 x 512] N(0,0.02); 512-pt Hadamard"),
    "llama2_7b": Workload(
        name="llama2_7b", T=2048, layers=_llama_layers(4096, 11008, 4096), x_dtype="bf16",
        dist="normal", n_out=4, mult=100.0, kv_heads=32,
        description="Llama-2-7B-shaped q/k/v/o/gate/up/down layers, hidden 4096, intermediate "
                    "11008, 2048 prefill tokens, bf16 N(0,1) + 4 outlier channels x100, "
                    "KV4 of 32 heads x 128"),
    "llama3_8b_mlp": Workload(
        name="llama3_8b_mlp", T=4096,
        layers=(Linear("gate", 4096, 14336, False), Linear("up", 4096, 14336, False),
                Linear("down", 14336, 4096, True)),
        x_dtype="bf16", dist="student_t3", n_out=3, mult=100.0,
        description="Llama-3-8B-shaped MLP 4096->14336 (gate/up), 14336->4096 (down, 14 x 1024 "
                    "blocks), 4096 prefill tokens, Student-t(3) + 3 outlier channels"),
    "llama2_70b": Workload(
        name="llama2_70b", T=8192, layers=_llama_layers(8192, 28672, 1024), x_dtype="bf16",
        dist="normal", n_out=6, mult=200.0, kv_heads=8,
        description="Llama-2-70B-shaped layers, hidden 8192, intermediate 28672, GQA 8 KV heads "
                    "x 128, 8192 prefill tokens, bf16 + 6 outlier channels x200"),
}

DECODE_BATCHES = (1, 8, 32, 64)


def decode_workload(T: int) -> Workload:
    return Workload(
        name=f"decode_t{T}", T=T, layers=(Linear("gate", 4096, 11008, False),), x_dtype="bf16",
        dist="normal", n_out=4, mult=100.0, kv_heads=32,
        description=f"decode on Llama-2-7B shapes: {T} tokens x 4096->11008 W4A4 linear + KV4 "
                    f"of 32 heads x 128 per token")


def layer_inputs(w: Workload, layer: Linear, T: Optional[int] = None, seed: int = SEED_X):
    """Activations for one layer of a workload as float32 numpy [T, K]."""
    T = w.T if T is None else T
    return activations(T, layer.K, seed=seed, dist=w.dist, n_out=w.n_out, mult=w.mult)
