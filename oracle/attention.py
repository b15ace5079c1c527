"""Tree-masked GQA attention over the reused prefix KV, in float64.

Section 3.2 ("Single-pass token verification"): one forward pass over the
current token and its proposal predicts a token at every proposed position.
Section 3.4 and Section 4 ("Runtime state management"): the prefix's K/V
states are carried forward in a cache and reused, so the verify pass
attends to the cached prefix plus the proposal itself.

For proposal node n and query head h (KV head g = h // G, G = Hq / Hkv):

    S(n)   = {prefix rows 0..P-1}  U  {tree rows i : i on the root path of n}
    s_j    = scale * <q[n, h], k_j>        for j in S(n)
    w_j    = exp(s_j - max s) / sum exp(s - max s)
    o[n,h] = sum_j w_j v_j

The root path is found by walking parent indices, not from any bitmap.
Queries and tree keys arrive already rotary-embedded (position P + depth).
"""
import math

import numpy as np

from .tree import ancestors_or_self


def tree_attention(q, prefix_k, prefix_v, tree_k, tree_v, parent, scale=None, nodes=None):
    """One sequence, one layer.

    q        [N, Hq, D]     queries of the N proposal nodes
    prefix_k [Hkv, P, D]    cached prefix keys   (P may be 0)
    prefix_v [Hkv, P, D]    cached prefix values
    tree_k   [N, Hkv, D]    keys of the proposal nodes
    tree_v   [N, Hkv, D]    values of the proposal nodes
    parent   [N]            parent[0] = -1
    scale    softmax scale, default 1/sqrt(D)
    nodes    optional subset of nodes to compute (others are left zero)
    returns  [N, Hq, D] float64
    """
    q = np.asarray(q, dtype=np.float64)
    prefix_k = np.asarray(prefix_k, dtype=np.float64)
    prefix_v = np.asarray(prefix_v, dtype=np.float64)
    tree_k = np.asarray(tree_k, dtype=np.float64)
    tree_v = np.asarray(tree_v, dtype=np.float64)
    N, Hq, D = q.shape
    Hkv = tree_k.shape[1]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(D)
    out = np.zeros((N, Hq, D), dtype=np.float64)
    for n in (range(N) if nodes is None else nodes):
        visible = sorted(ancestors_or_self(parent, n))
        for h in range(Hq):
            g = h // G
            keys = np.concatenate([prefix_k[g], tree_k[visible, g, :]], axis=0)
            vals = np.concatenate([prefix_v[g], tree_v[visible, g, :]], axis=0)
            s = (keys @ q[n, h]) * scale
            w = np.exp(s - s.max())
            w = w / w.sum()
            out[n, h] = w @ vals
    return out
