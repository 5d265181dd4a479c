"""O2: rotary position embedding, rotate-half form (fp64).

The paper runs every configuration inside Hugging Face Transformers on Llama
3.1 8B (Section 2.3, Section 3.1), whose attention uses the rotate-half
rotary embedding: channel i is paired with channel i + D/2, and the pair is
rotated by the angle p * omega_i with omega_i = theta^(-2i/D).

    x'_i       = x_i cos(p w_i) - x_{i+D/2} sin(p w_i)
    x'_{i+D/2} = x_{i+D/2} cos(p w_i) + x_i sin(p w_i)

KVQuant quantizes keys before this rotation, so the decode path rotates each
dequantized key by its position (Section 2.1, KVQuant paragraph).
"""
from __future__ import annotations

import numpy as np


def inv_freq(D: int, theta: float) -> np.ndarray:
    """omega_i = theta^(-2i/D), i < D/2, float64."""
    i = np.arange(D // 2, dtype=np.float64)
    return np.power(float(theta), -2.0 * i / D)


def apply(x, positions, theta: float):
    """Rotate rows ``x`` [..., n, D] at integer ``positions`` [n]."""
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    ang = np.asarray(positions, dtype=np.float64)[:, None] * inv_freq(D, theta)[None, :]
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., : D // 2], x[..., D // 2:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)
