"""Scalar numerics of the LLaMA-style decoder (fp64).

The paper names LLaMA-7B as the target backbone (Sec. 4.1) but fixes no
constants; the readings used here are RMSNorm with eps 1e-6, RoPE with
theta 1e4 and rotate-half pairing (i, i + hd/2), SiLU-gated MLP, no biases.
"""
from __future__ import annotations

import numpy as np


def bf16(x) -> np.ndarray:
    """Round to the nearest bfloat16 value (8 significant bits, ties to even), in fp64.

    With x = m * 2**e and 0.5 <= |m| < 1, a bf16 value keeps 8 significant bits,
    i.e. round(m * 2**8) * 2**(e - 8); ``np.rint`` rounds half to even.
    """
    x = np.asarray(x, dtype=np.float64)
    m, e = np.frexp(x)
    return np.ldexp(np.rint(m * 256.0), e - 8)


def rms_scale(h: np.ndarray, eps: float) -> np.ndarray:
    """RMSNorm's per-row scale 1 / sqrt(mean(h^2) + eps) over the last axis (keepdims)."""
    h = np.asarray(h, dtype=np.float64)
    return 1.0 / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps)


def rmsnorm(h: np.ndarray, g: np.ndarray, eps: float) -> np.ndarray:
    """h / sqrt(mean(h^2) + eps) * g over the last axis."""
    h = np.asarray(h, dtype=np.float64)
    ms = np.mean(h * h, axis=-1, keepdims=True)
    return h / np.sqrt(ms + eps) * np.asarray(g, dtype=np.float64)


def rope_angles(pos: np.ndarray, head_dim: int, theta: float) -> np.ndarray:
    """angle[t, i] = pos[t] * theta**(-2i/hd) for i < hd/2."""
    i = np.arange(head_dim // 2, dtype=np.float64)
    inv = theta ** (-2.0 * i / head_dim)
    return np.asarray(pos, dtype=np.float64)[:, None] * inv[None, :]


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing: x has shape [T, H, hd]."""
    hd = x.shape[-1]
    half = hd // 2
    ang = rope_angles(pos, hd, theta)[:, None, :]       # [T, 1, hd/2]
    c, s = np.cos(ang), np.sin(ang)
    a, b = x[..., :half], x[..., half:]
    return np.concatenate([a * c - b * s, b * c + a * s], axis=-1)


def silu(x: np.ndarray) -> np.ndarray:
    return x / (1.0 + np.exp(-x))


def softmax(x: np.ndarray, axis: int = -1) -> np.ndarray:
    m = np.max(x, axis=axis, keepdims=True)
    e = np.exp(x - m)
    return e / np.sum(e, axis=axis, keepdims=True)
