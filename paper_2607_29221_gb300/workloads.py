"""Seeded synthetic inputs and workload shapes.

This module is shared by the CUDA path, the oracle and the benchmark, so it
holds none of the method's arithmetic: only random floating-point inputs drawn
from numpy's PCG64 generator, the 256-bit mask key, and the matrix shapes of the
transformer workloads the paper evaluates (Sec. 5 and Fig. 1: LLaMA/Qwen 7B and
70B-class projections).  The paper's weights and datasets (WikiText-2,
HumanEval, model checkpoints) are not available; Gaussian matrices of the same
shapes stand in for them: activations ~ N(0, 1), weights ~ N(0, 0.02) (N(0, 1)
for the small case).

All matrices are returned token-major / row-major float32:
  X_tm : l x n   (token k is row k; the paper's X is n x l, i.e. X_tm = X^T)
  W    : m x n   (the paper's weight matrix, output row j is row j)
"""
from __future__ import annotations

import hashlib
from dataclasses import dataclass, field

import numpy as np

# Seeds for the two float inputs of every workload.
SEED_X = 1
SEED_W = 2
# Bias of the linear layer is drawn from its own seed (Pi_Sec-Linear input b).
SEED_B = 3


def mask_key() -> np.ndarray:
    """256-bit PRG key as 8 little-endian uint32 words: SHA-256 of a fixed label."""
    digest = hashlib.sha256(b"MOSAIC-2607.29221").digest()
    return np.frombuffer(digest, dtype="<u4").astype(np.uint32).copy()


def gaussian_f32(seed: int, rows: int, cols: int, std: float) -> np.ndarray:
    """rows x cols float32 ~ N(0, std^2) from PCG64(seed)."""
    g = np.random.Generator(np.random.PCG64(seed))
    a = g.standard_normal((rows, cols), dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return a


def gaussian_f32_rows(seed: int, rows: int, cols: int, std: float, which) -> np.ndarray:
    """Rows `which` (ascending) of gaussian_f32(seed, rows, cols, std), drawn in
    chunks so that the whole matrix is never held at once."""
    which = np.asarray(which, dtype=np.int64)
    g = np.random.Generator(np.random.PCG64(seed))
    out = np.empty((len(which), cols), np.float32)
    chunk = max(1, (1 << 24) // max(cols, 1))
    start, k = 0, 0
    while start < rows and k < len(which):
        n = min(chunk, rows - start)
        a = g.standard_normal((n, cols), dtype=np.float32)
        while k < len(which) and which[k] < start + n:
            out[k] = a[which[k] - start]
            k += 1
        start += n
    if std != 1.0:
        out *= np.float32(std)
    return out


def activations(l: int, n: int, seed: int = SEED_X, std: float = 1.0) -> np.ndarray:
    return gaussian_f32(seed, l, n, std)


def weights(m: int, n: int, seed: int = SEED_W, std: float = 0.02) -> np.ndarray:
    return gaussian_f32(seed, m, n, std)


def weight_rows(m: int, n: int, which, seed: int = SEED_W, std: float = 0.02) -> np.ndarray:
    """Rows `which` (ascending) of weights(m, n, seed, std)."""
    return gaussian_f32_rows(seed, m, n, std, which)


def bias(m: int, seed: int = SEED_B, std: float = 0.02) -> np.ndarray:
    return gaussian_f32(seed, 1, m, std)[0]


def spike_activations(l: int, n: int, seed: int = SEED_X, outlier: float = 100.0,
                      channels: int = 4) -> np.ndarray:
    """N(0,1) activations with a few outlier channels (100x), the activation
    structure Sec. 4 describes for transformer layers."""
    a = activations(l, n, seed)
    g = np.random.Generator(np.random.PCG64(seed + 1000))
    ch = g.choice(n, size=channels, replace=False)
    a[:, ch] *= np.float32(outlier)
    return a


def outlier_weights(m: int, n: int, seed: int = SEED_W, std: float = 0.02, channels: int = 8,
                    factor: float = 10.0) -> np.ndarray:
    """N(0, std^2) weights whose few input channels (columns) are `factor`
    times larger: the outlier-channel structure of trained LLM projections
    that the rotation of Sec. 4 spreads out."""
    w = weights(m, n, seed, std)
    g = np.random.Generator(np.random.PCG64(seed + 2000))
    ch = g.choice(n, size=channels, replace=False)
    w[:, ch] *= np.float32(factor)
    return w


def uniform_u32(seed: int, rows: int, cols: int) -> np.ndarray:
    """Uniform ring elements for ring-only tests (not part of the protocol's PRG)."""
    g = np.random.Generator(np.random.PCG64(seed))
    return g.integers(0, 1 << 32, size=(rows, cols), dtype=np.uint32)


@dataclass(frozen=True)
class Linear:
    """One outsourced linear layer: W is m x n, applied to l tokens."""
    name: str
    m: int
    n: int
    w_std: float = 0.02


@dataclass(frozen=True)
class Workload:
    name: str
    l: int                       # tokens per pass
    linears: tuple               # tuple[Linear, ...]
    x_std: float = 1.0
    notes: str = ""
    decode_batches: tuple = field(default=())


# Shapes of the transformer workloads the paper measures (7B and 70B-class
# layers, Sec. 5), plus a small case the oracle finishes in well under a second.
WORKLOADS = {
    "single_64x256x128": Workload(
        "single_64x256x128", 64, (Linear("w", 128, 256, 1.0),),
        notes="X 64x256, W 256->128, both N(0,1); rotation dim 256"),
    "attn_proj_7b_512x4096x4096": Workload(
        "attn_proj_7b_512x4096x4096", 512, (Linear("attn", 4096, 4096),),
        notes="attention projection at 7B shape; rotation dim 4096"),
    "ffn_7b_2048x4096x14336": Workload(
        "ffn_7b_2048x4096x14336", 2048,
        (Linear("up", 14336, 4096), Linear("down", 4096, 14336)),
        notes="FFN up and down at 7B shape; rotation dims 4096 and 16384 (14336 padded)"),
    "decoder_70b_prefill_2048": Workload(
        "decoder_70b_prefill_2048", 2048,
        (Linear("qkv", 10240, 8192), Linear("o", 8192, 8192),
         Linear("gate_up", 57344, 8192), Linear("down", 8192, 28672)),
        notes="one 70B decoder layer, 64 q / 8 kv heads, head dim 128, SwiGLU 28672"),
    "decode_70b_sweep": Workload(
        "decode_70b_sweep", 1,
        (Linear("qkv", 9216, 8192), Linear("qkv10240", 10240, 8192), Linear("o", 8192, 8192),
         Linear("gate_up", 57344, 8192), Linear("down", 8192, 28672)),
        decode_batches=(1, 8, 32, 128, 256),
        notes="decode sweep at 70B layer shape, pre-masked weights"),
    "matvec_sweep": Workload(
        "matvec_sweep", 1,
        (Linear("n4096", 4096, 4096), Linear("n8192", 8192, 8192), Linear("n16384", 16384, 16384),
         Linear("n36864", 36864, 36864)),
        notes="secure mat-vec n x n, one token (the paper's mat-vec figure; n = 36864 is "
              "rotated at width 65536)"),
    "sigma_sweep_7b": Workload(
        "sigma_sweep_7b", 128,
        (Linear("attn", 4096, 4096), Linear("up", 14336, 4096), Linear("down", 4096, 14336)),
        notes="single-layer relative l2 error vs sigma (the paper's single-layer error table), "
              "N(0,0.02) weights with 8 outlier input channels (10x), N(0,1) activations with "
              "4 outlier channels (20x)"),
    "kernels_hbm": Workload(
        "kernels_hbm", 2048,
        (Linear("n4096", 4096, 4096), Linear("n16384", 4096, 16384), Linear("n32768", 1024, 32768)),
        notes="memory-bound client kernels alone (rotation, encode + mask-add (+ digit planes), "
              "E_x sampling) on token batches of l x n_pad, L2 flushed between launches"),
    "init_w_70b": Workload(
        "init_w_70b", 0,
        (Linear("qkv", 10240, 8192), Linear("o", 8192, 8192),
         Linear("gate_up", 57344, 8192), Linear("down", 8192, 28672)),
        notes="one-time Init W of a 70B layer's four matrices plus the public chains per "
              "rotation width, extrapolated to 80 layers"),
}

