"""Rotary position embedding (RoPE) of q and k, plain fp64 on the CPU.

TEST INFRASTRUCTURE ONLY: imported by tests/, __graft_entry__.smoke() and the
CPU-baseline / reference legs of bench.py. The CUDA path never imports it, and
it imports nothing from the CUDA path.

The model section of the paper (Sec. 3, training setup) places RoPE before the
attention module: consecutive components of every query and key head vector are
rotated, with base frequency f_b (10k by default; 100k in the curriculum and
scaling runs, Table 2 and the f_b ablation table). Written out:

    position m of a token = its index inside its sequence (0 .. L-1)
    theta_j = f_b ** (-2 j / d),             j = 0 .. d/2 - 1
    (x[2j], x[2j+1]) -> (x[2j] cos(m theta_j) - x[2j+1] sin(m theta_j),
                         x[2j] sin(m theta_j) + x[2j+1] cos(m theta_j))

The rotation R_m is orthogonal, so the gradient with respect to the
un-rotated vector is R_m^T applied to the gradient with respect to the rotated
one. Training runs in bf16 (Sec. 3), so the attention consumes the rotated q
and k rounded to bf16 (`round_to_bf16`).
"""
from __future__ import annotations

import numpy as np


def angles(L: int, d: int, base: float) -> np.ndarray:
    """[L, d/2] rotation angles m * theta_j in float64."""
    j = np.arange(d // 2, dtype=np.float64)
    theta = np.power(float(base), -2.0 * j / d)
    m = np.arange(L, dtype=np.float64)
    return m[:, None] * theta[None, :]


def rope_rotate(x: np.ndarray, base: float) -> np.ndarray:
    """x: [B, L, H, d] float64 -> R_m x for every token (pairs of consecutive components)."""
    B, L, H, d = x.shape
    a = angles(L, d, base)[None, :, None, :]           # [1, L, 1, d/2]
    c, s = np.cos(a), np.sin(a)
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x, dtype=np.float64)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def rope_unrotate(g: np.ndarray, base: float) -> np.ndarray:
    """R_m^T g: the gradient with respect to the un-rotated vectors."""
    B, L, H, d = g.shape
    a = angles(L, d, base)[None, :, None, :]
    c, s = np.cos(a), np.sin(a)
    g0, g1 = g[..., 0::2], g[..., 1::2]
    out = np.empty_like(g, dtype=np.float64)
    out[..., 0::2] = g0 * c + g1 * s
    out[..., 1::2] = -g0 * s + g1 * c
    return out


def round_to_bf16(x: np.ndarray) -> np.ndarray:
    """Round float64 values to the nearest bfloat16 value (8 significant bits,
    ties to even, exponent range of float32 with subnormals), returned as
    float64."""
    x = np.asarray(x, dtype=np.float64)
    mant, exp = np.frexp(x)                      # x = mant * 2**exp, 0.5 <= |mant| < 1
    # spacing of bf16 values near x: 2**(exp - 8) for normals, 2**-133 below 2**-126
    q_exp = np.maximum(exp - 8, -133)
    return np.ldexp(np.rint(np.ldexp(x, -q_exp)), q_exp)
