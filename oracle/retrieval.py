"""Decoding-experience retrieval: token-filtered cosine top-1 over int8 keys.

Section 3.2 ("Context-compatible retrieval"): a query is the pair (h_i, y_i)
of the current final-layer state and token.  The search is restricted to
stored entries (h_j, p_j, b_j) whose token at position p_j equals y_i and
for which p_j < b_j (a proposal must not cross the stored output's
boundary); among them the entry whose key has the highest cosine
similarity with the query's is selected, with that similarity as s.
Section 4 ("Memory and retrieval"): keys are 256-dimensional int8 vectors
obtained from the normalised final-layer state by a fixed random
projection.

Readings (the paper does not fix them): the int8 code of a projected vector
z is round-half-to-even(127 * z / max|z|) (cosine is scale invariant, so a
per-vector scale keeps every key at full int8 resolution); ties in
similarity go to the lowest entry index; entries whose key is all zero have
no defined cosine and are never selected; no eligible entry -> index -1.
"""
import math

import numpy as np


def project_key(h, proj):
    """h [H] (final-layer state), proj [256, H] -> (int8 key [256], the
    pre-rounding values 127 * z / max|z| [256] float64)."""
    h = np.asarray(h, dtype=np.float64)
    hn = h / np.linalg.norm(h)
    z = np.asarray(proj, dtype=np.float64) @ hn
    x = 127.0 * z / np.max(np.abs(z))
    return np.rint(x).astype(np.int8), x   # numpy rint: round half to even


def _better(dot_a, kk_a, dot_b, kk_b):
    """Is dot_a / sqrt(kk_a) > dot_b / sqrt(kk_b)?  Exact, on Python ints."""
    if (dot_a >= 0) != (dot_b >= 0):
        return dot_a >= 0
    lhs, rhs = dot_a * dot_a * kk_b, dot_b * dot_b * kk_a
    return lhs > rhs if dot_a >= 0 else lhs < rhs


def cosine_top1(qkey, keys, entry_token, entry_pos, entry_bound, token, lo=0, hi=None):
    """Scan entries [lo, hi): returns (best index or -1, cosine similarity or nan)."""
    keys = np.asarray(keys)
    hi = len(keys) if hi is None else hi
    q = [int(v) for v in qkey]
    qq = sum(v * v for v in q)
    best, best_dot, best_kk = -1, 0, 1
    for j in range(lo, hi):
        if int(entry_token[j]) != int(token) or not int(entry_pos[j]) < int(entry_bound[j]):
            continue
        k = [int(v) for v in keys[j]]
        kk = sum(v * v for v in k)
        if kk == 0:
            continue
        dot = sum(a * b for a, b in zip(q, k))
        if best < 0 or _better(dot, kk, best_dot, best_kk):
            best, best_dot, best_kk = j, dot, kk
    if best < 0:
        return -1, float("nan")
    return best, best_dot / math.sqrt(qq * best_kk)
