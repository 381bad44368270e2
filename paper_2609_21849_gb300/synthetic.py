"""Seeded synthetic inputs for the quantized linear layer.

The paper measures the FLUX.2-klein denoiser at 1024x1024 (4096 image tokens
+ 512 text tokens; hidden 3072, MLP 12288) and its 0.6B->4B embedding
translator (1024 <-> 2560), Sec. 3 and Sec. 4.  Neither the checkpoints nor the
prompt set are available, so these generators stand in for them with random
activations and weights of the same shapes and value structure.

This module holds no arithmetic of the method: it draws numbers (numpy PCG64)
and rounds them to bf16 (round to nearest even) so that the CUDA path and the
CPU oracle see identical bits.  Both sides take their inputs from here.

Recipes (seed s):
  * activations: rng = default_rng(s); z ~ N(0, 1) in fp32.
      - "entry outliers": round(0.01 * M * K) entries, chosen uniformly
        without replacement, are multiplied by 20.
      - "channel gain": x = z * g[k], g = exp(N(0, 1)) per channel k.
      - "channel outliers": round(0.01 * K) channels multiplied by 20.
  * weights: rng = default_rng([s, 1]) (the translator MLP: [s, 3]);
    w ~ N(0, sigma^2), drawn in the order the weights are listed.
"""
from __future__ import annotations

import numpy as np

# Shapes of the five workloads (M, K, N), named for what they are.
M_TOKENS = 4608          # 4096 image tokens + 512 text tokens at 1024x1024
HIDDEN = 3072
MLP = 12288


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to bf16 (nearest, ties to even); return uint16 bits.
    Inputs are finite."""
    a = np.ascontiguousarray(a, np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = (u + 0x7FFF + lsb) >> 16
    return r.astype(np.uint16)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(bits, np.uint16).astype(np.uint32) << 16).view(np.float32)


def _normal(rng, shape, sigma=1.0):
    z = rng.standard_normal(shape, dtype=np.float32)
    if sigma != 1.0:
        z *= np.float32(sigma)
    return z


def act_entry_outliers(seed: int, M: int, K: int, frac=0.01, gain=20.0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    x = _normal(rng, (M, K))
    n = int(round(frac * M * K))
    idx = rng.choice(M * K, size=n, replace=False)
    x.reshape(-1)[idx] *= np.float32(gain)
    return bf16_bits(x)


def act_channel_gain(seed: int, M: int, K: int, sigma=1.0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    z = _normal(rng, (M, K))
    g = np.exp(rng.standard_normal(K) * sigma).astype(np.float32)
    return bf16_bits(z * g[None, :])


def act_channel_outliers(seed: int, M: int, K: int, frac=0.01, gain=20.0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    x = _normal(rng, (M, K))
    n = int(round(frac * K))
    ch = rng.choice(K, size=n, replace=False)
    x[:, ch] *= np.float32(gain)
    return bf16_bits(x)


def act_normal(seed: int, M: int, K: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    return bf16_bits(_normal(rng, (M, K)))


def weights(seed: int, shapes, sigma: float, stream: int = 1):
    """Weights [N, K] ~ N(0, sigma^2) for each (N, K) in ``shapes``, drawn in
    order from default_rng([seed, stream]).  Yields bf16 bit arrays."""
    rng = np.random.default_rng([seed, stream])
    for (N, K) in shapes:
        yield bf16_bits(_normal(rng, (N, K), sigma))


# ------------------------------------------------------------- workloads ---

def tiny_nvfp4(M=128, K=256, N=256, seed=0):
    """NVFP4 W4A4 linear, tiny (128x256 by 256x256), entry outliers."""
    x = act_entry_outliers(seed, M, K)
    (w,) = weights(seed, [(N, K)], 0.02)
    return x, w


def fp8_linear(M=M_TOKENS, K=HIDDEN, N=HIDDEN, seed=1):
    """FP8 linear at the denoiser's hidden size, log-normal channel gains."""
    x = act_channel_gain(seed, M, K)
    (w,) = weights(seed, [(N, K)], 0.02)
    return x, w


def nvfp4_mlp_up(M=M_TOKENS, K=HIDDEN, N=MLP, seed=2):
    """NVFP4 MLP up-projection (4608x3072 by 12288x3072), entry outliers."""
    x = act_entry_outliers(seed, M, K)
    (w,) = weights(seed, [(N, K)], 0.02)
    return x, w


def translator(M=512, seed=3):
    """Translator-shaped small-M linears (batch 1, 512 tokens): x1 [512, 1024]
    feeds W1 [2560, 1024]; x2 [512, 2560] feeds W2 [1024, 2560]; activations
    N(0, 1) (x2 from default_rng([seed, 2])), weights N(0, 0.03^2)."""
    x1 = act_normal(seed, M, 1024)
    x2 = bf16_bits(_normal(np.random.default_rng([seed, 2]), (M, 2560)))
    w1, w2 = weights(seed, [(2560, 1024), (1024, 2560)], 0.03)
    return x1, x2, w1, w2


TRANSLATOR_IN, TRANSLATOR_HIDDEN, TRANSLATOR_OUT = 1024, 3072, 2560


def translator_mlp(M=512, seed=3):
    """The d3072 translator MLP (0.6B encoder features -> 4B conditioning):
    x [512, 1024] N(0, 1) (the translator linears' x1), W1 [3072, 1024] and
    W2 [2560, 3072] N(0, 0.03^2) from default_rng([seed, 3])."""
    x = act_normal(seed, M, TRANSLATOR_IN)
    w1, w2 = weights(seed, [(TRANSLATOR_HIDDEN, TRANSLATOR_IN),
                            (TRANSLATOR_OUT, TRANSLATOR_HIDDEN)], 0.03, stream=3)
    return x, w1, w2


STACK_LAYERS = (("qkv", 3 * HIDDEN, HIDDEN), ("out", HIDDEN, HIDDEN),
                ("up", MLP, HIDDEN), ("down", HIDDEN, MLP))


def stack_input(B=1, seed=4):
    """Input of the denoise-step linear stack: [4608*B, 3072], channel
    outliers (1% of channels x20)."""
    return act_channel_outliers(seed, M_TOKENS * B, HIDDEN)


def stack_weights(n_blocks=8, seed=4):
    """Yields (block, name, bf16 bits [N, K]) for the stack's 8 x 4 linears."""
    shapes = [(N, K) for _ in range(n_blocks) for (_, N, K) in STACK_LAYERS]
    names = [(b, name) for b in range(n_blocks) for (name, _, _) in STACK_LAYERS]
    for (b, name), w in zip(names, weights(seed, shapes, 0.02)):
        yield b, name, w
