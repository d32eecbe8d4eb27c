"""Seeded synthetic inputs shaped like the paper's DiT / UNet linear layers.

This module is shared by the CPU oracle tests, the GPU parity tests and the
benchmark.  It holds only input generation (random draws, casts to fp16,
im2col re-indexing); none of the quantizer's or the GEMM's arithmetic lives
here.  Every tensor is a NumPy array of dtype float16 generated on the CPU
from ``numpy.random.default_rng(seed)`` so that both sides of a parity test
receive identical bits.

The paper's datasets and trained weights (LSUN, CelebA-HQ, FFHQ, MS-COCO,
MJHQ-30K, sDCI; LDM, SD, PixArt-Sigma, FLUX.1-schnell checkpoints) are not
available; these recipes stand in for them:

* activations: Laplace(0, 0.05) bulk with a seeded subset of channels
  (columns of K) scaled up to mimic per-channel outliers (Section 1 and
  Section 3 motivate LSB-dense activations plus sparse outliers);
* weights: N(0, 0.02) in fp16, the usual DiT/UNet initialisation scale;
* the encode sweep: an i.i.d. mixture 89% Laplace(0,0.05), 10% N(0,0.3),
  1% U(-8,8);
* UNet convolutions: SiLU(N(0,1)) feature maps with sparse x10 channels,
  lowered to a GEMM by im2col with K ordered (kh, kw, c_in), padding 1;
* attention decode step (Appendix D, Table 6): N(0, 1) queries, keys and
  values, 2% of the key dimensions x8;
* LLM layers (Section 5 variant; the paper's Qwen2 / LLaMA checkpoints and
  its perplexity corpus are not available): the Laplace recipe with 0.2% of
  the channels x100, the few very large channels of LLM hidden states.
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

BASE_SEED = 2509_26436


def seed_for(config: int, layer: int, role: int = 0) -> int:
    """Seed of (config, layer, role); role 0 = activations, 1 = weights."""
    return BASE_SEED + 1000 * config + 10 * layer + role


def _outlier_channels(rng: np.random.Generator, K: int, frac: float) -> np.ndarray:
    n = max(1, int(round(K * frac))) if frac > 0 else 0
    return rng.permutation(K)[:n]


def laplace_activations(M: int, K: int, seed: int, b: float = 0.05,
                        outlier_frac: float = 0.005, outlier_scale: float = 20.0) -> np.ndarray:
    """Laplace(0, b) activations [M, K] with `outlier_frac` of the K channels
    multiplied by `outlier_scale` (seeded permutation), cast to fp16."""
    rng = np.random.default_rng(seed)
    x = rng.laplace(0.0, b, size=(M, K)).astype(np.float32)
    ch = _outlier_channels(rng, K, outlier_frac)
    if ch.size:
        x[:, ch] *= np.float32(outlier_scale)
    return x.astype(np.float16)


def mixture_activations(rows: int, K: int, seed: int) -> np.ndarray:
    """Encode-sweep mixture [rows, K]: per element 89% Laplace(0,0.05),
    10% N(0,0.3), 1% U(-8,8); fp16."""
    rng = np.random.default_rng(seed)
    u = rng.random(size=(rows, K), dtype=np.float32)
    lap = rng.laplace(0.0, 0.05, size=(rows, K)).astype(np.float32)
    gau = rng.normal(0.0, 0.3, size=(rows, K)).astype(np.float32)
    uni = rng.uniform(-8.0, 8.0, size=(rows, K)).astype(np.float32)
    x = np.where(u < 0.89, lap, np.where(u < 0.99, gau, uni))
    return x.astype(np.float16)


def gaussian_weights(N: int, K: int, seed: int, std: float = 0.02) -> np.ndarray:
    """nn.Linear-layout weights [N, K] ~ N(0, std), fp16."""
    rng = np.random.default_rng(seed)
    return rng.normal(0.0, std, size=(N, K)).astype(np.float32).astype(np.float16)


def silu_im2col(batch: int, C: int, H: int, W: int, seed: int,
                outlier_frac: float = 0.005, outlier_scale: float = 10.0) -> np.ndarray:
    """3x3 / stride 1 / pad 1 convolution input lowered to a GEMM operand.

    x[b, c, h, w] = SiLU(N(0,1)) with `outlier_frac` of the input channels
    scaled by `outlier_scale`; returns A [batch*H*W, 9*C] fp16 with K ordered
    (kh, kw, c).  Zero padding produces exactly-zero K groups at the borders.
    """
    rng = np.random.default_rng(seed)
    z = rng.normal(0.0, 1.0, size=(batch, C, H, W)).astype(np.float32)
    x = z / (1.0 + np.exp(-z))
    ch = _outlier_channels(rng, C, outlier_frac)
    if ch.size:
        x[:, ch] *= np.float32(outlier_scale)
    x16 = x.astype(np.float16)
    xp = np.zeros((batch, C, H + 2, W + 2), dtype=np.float16)
    xp[:, :, 1:H + 1, 1:W + 1] = x16
    cols = np.empty((batch, H, W, 3, 3, C), dtype=np.float16)
    for kh in range(3):
        for kw in range(3):
            # [batch, C, H, W] window -> [batch, H, W, C]
            cols[:, :, :, kh, kw, :] = xp[:, :, kh:kh + H, kw:kw + W].transpose(0, 2, 3, 1)
    return cols.reshape(batch * H * W, 9 * C)


@dataclass(frozen=True)
class Layer:
    """One W4A4 linear: activations [M, K] times weights [N, K]^T."""
    name: str
    M: int
    N: int
    K: int
    config: int
    index: int
    kind: str = "laplace"          # laplace | conv
    outlier_frac: float = 0.005
    outlier_scale: float = 20.0
    conv: tuple | None = None      # (batch, C, H, W) for kind == "conv"

    @property
    def ops(self) -> int:
        return 2 * self.M * self.N * self.K

    def activations(self) -> np.ndarray:
        s = seed_for(self.config, self.index, 0)
        if self.kind == "conv":
            b, c, h, w = self.conv
            return silu_im2col(b, c, h, w, s, self.outlier_frac, self.outlier_scale)
        return laplace_activations(self.M, self.K, s, 0.05, self.outlier_frac, self.outlier_scale)

    def weights(self) -> np.ndarray:
        return gaussian_weights(self.N, self.K, seed_for(self.config, self.index, 1))


# Single W4A4 linear, 256 tokens x 1152 hidden (small enough for the oracle).
CONFIG0 = [Layer("single_1152", 256, 1152, 1152, 0, 0)]

# PixArt-Sigma block linears at 1024px: 4096 image tokens x batch 2, hidden 1152.
CONFIG2 = [
    Layer("pixart_qkv", 8192, 3456, 1152, 2, 0),
    Layer("pixart_proj", 8192, 1152, 1152, 2, 1),
    Layer("pixart_fc1", 8192, 4608, 1152, 2, 2),
    Layer("pixart_fc2", 8192, 1152, 4608, 2, 3),
]

# SDXL UNet 3x3 convolutions as im2col GEMMs, batch 2, K = 9 * C_in.
CONFIG3 = [
    Layer("sdxl_conv1280_32x32", 2 * 32 * 32, 1280, 9 * 1280, 3, 0, kind="conv",
          outlier_frac=0.005, outlier_scale=10.0, conv=(2, 1280, 32, 32)),
    Layer("sdxl_conv640_64x64", 2 * 64 * 64, 640, 9 * 640, 3, 1, kind="conv",
          outlier_frac=0.005, outlier_scale=10.0, conv=(2, 640, 64, 64)),
]

# FLUX.1-schnell MM-DiT block linears: (4096 + 512) tokens x batch 4, hidden 3072.
CONFIG4 = [
    Layer("flux_qkv", 18432, 9216, 3072, 4, 0, outlier_frac=0.001, outlier_scale=50.0),
    Layer("flux_proj", 18432, 3072, 3072, 4, 1, outlier_frac=0.001, outlier_scale=50.0),
    Layer("flux_fc1", 18432, 12288, 3072, 4, 2, outlier_frac=0.001, outlier_scale=50.0),
    Layer("flux_fc2", 18432, 3072, 12288, 4, 3, outlier_frac=0.001, outlier_scale=50.0),
]

# LLaMA-2-7B decoder block linears (Section 5 LLM variant, 16-bit codes,
# G_s = 8) at a 2048-token prefill: hidden 4096, MLP 11008 (gate and up
# fused), activations with a few strong outlier channels.
CONFIG_LLM = [
    Layer("llama2_qkv", 2048, 12288, 4096, 5, 0, outlier_frac=0.002, outlier_scale=100.0),
    Layer("llama2_o", 2048, 4096, 4096, 5, 1, outlier_frac=0.002, outlier_scale=100.0),
    Layer("llama2_gate_up", 2048, 22016, 4096, 5, 2, outlier_frac=0.002, outlier_scale=100.0),
    Layer("llama2_down", 2048, 4096, 11008, 5, 3, outlier_frac=0.002, outlier_scale=100.0),
]

# Attention decode step (Appendix D, Table 6: heads x 128 dimensions, LZS
# groups 8 / 16 / 32): batch 16, a 4096-token key / value cache per head.
ATTN_HEADS = (32, 40, 64)
ATTN_DIM = 128
ATTN_BATCH = 16
ATTN_CONTEXT = 4096


def attention_inputs(BH: int, L: int, seed: int, outlier_frac: float = 0.02, outlier_scale: float = 8.0):
    """q [BH, 128], k and v [BH * L, 128] fp16 (head bh's tokens in rows
    bh * L ..): N(0, 1) entries, the keys with a seeded `outlier_frac` of the
    head dimensions scaled by `outlier_scale` (the outlier channels of LLM
    keys), the queries and values plain."""
    rng = np.random.default_rng(seed)
    d = ATTN_DIM
    q = rng.normal(0.0, 1.0, size=(BH, d)).astype(np.float32)
    k = rng.normal(0.0, 1.0, size=(BH * L, d)).astype(np.float32)
    ch = _outlier_channels(rng, d, outlier_frac)
    if ch.size:
        k[:, ch] *= np.float32(outlier_scale)
    v = rng.normal(0.0, 1.0, size=(BH * L, d)).astype(np.float32)
    return q.astype(np.float16), k.astype(np.float16), v.astype(np.float16)


# Encode sweep sizes: 1M, 16M and 128M fp16 elements as [rows, 4096].
ENCODE_SWEEP = [(2 ** 20 // 4096, 4096), (4096, 4096), (32768, 4096)]

GEMM_CONFIGS = {0: CONFIG0, 2: CONFIG2, 3: CONFIG3, 4: CONFIG4, 5: CONFIG_LLM}
