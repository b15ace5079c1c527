"""Rolling-image KV carryover: re-rotating cached keys to new positions.

Section 3.4 ("Rolling-image KV-state carryover"): when a multi-image window
advances, each retained screenshot's visual-token block moves to a new span
of the prompt.  Its cached keys, rotary-embedded at position m, are carried
to position m' by K~(m') = R(m') R(m)^-1 K~(m); its values are reused
unchanged.  R(m) is the model's rotary position embedding at position m.

Rotary embedding used here (the rotate-half layout of the Qwen/Llama
families): for a head of dimension D and frequency index i < D/2 with
theta_i = base^(-2i/D), the pair (x_i, x_{i+D/2}) is rotated by the angle
m * theta_i.  For multi-axis rotary embeddings (image tokens with temporal,
height and width position components), moving a block shifts every
component by the same amount, so every frequency again turns by the same
multiple of the shift; R(m') R(m)^-1 therefore acts as below for them too.
"""
import numpy as np


def frequencies(D, base):
    return base ** (-2.0 * np.arange(D // 2, dtype=np.float64) / D)


def rotate(x, position, base):
    """R(position) applied to vectors x [..., D] (rotate-half layout), float64."""
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    ang = float(position) * frequencies(D, base)
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., : D // 2], x[..., D // 2:]
    return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)


def carry_keys(k_rot, m, m_new, base):
    """K~(m') = R(m') R(m)^-1 K~(m) for keys k_rot [..., D] rotated at m."""
    return rotate(rotate(k_rot, -m, base), m_new, base)


def shift_block(cache_k, cache_v, src, dst, n, base):
    """Move a block of n cached rows from positions src.. to dst.. of one
    sequence's cache rows [Hkv, S, D]: keys re-rotated from position p to
    p + (dst - src), values copied.  Returns new (K, V) copies; rows outside
    the destination span keep their old contents (a left move leaves the
    vacated tail as it was)."""
    K = np.array(cache_k, dtype=np.float64, copy=True)
    V = np.array(cache_v, dtype=np.float64, copy=True)
    src_k = np.array(cache_k[:, src:src + n, :], dtype=np.float64)
    src_v = np.array(cache_v[:, src:src + n, :], dtype=np.float64)
    for j in range(n):
        K[:, dst + j, :] = carry_keys(src_k[:, j, :], src + j, dst + j, base)
        V[:, dst + j, :] = src_v[:, j, :]
    return K, V
