"""Carry-forward of the accepted rows' K/V into the cache.

Section 1 and Section 3.4: accepted positions keep their K/V states so the
next step reuses them; Section 4 keeps one contiguous cache.  The root (the
current token, not yet cached) and the a accepted drafts become cache rows
P .. P + a; rejected proposal rows are discarded.  Row k of the accepted
path sits at position P + k = P + depth(path[k]), the position its key was
rotary-embedded at, so the rows move unchanged.
"""
import numpy as np


def commit_rows(cache_rows, prefix_len, path, tree_rows):
    """cache_rows [Hkv, S, D] of one sequence and layer (K or V),
    tree_rows [N, Hkv, D]; returns (new cache copy, new length)."""
    out = np.array(cache_rows, copy=True)
    for k, node in enumerate(path):
        out[:, prefix_len + k, :] = tree_rows[node, :, :]
    return out, prefix_len + len(path)
