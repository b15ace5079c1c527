"""Proposal-tree structure, by walking parent indices.

A proposal tree has node 0 = the current token (the root, whose K/V is not
yet cached) and nodes 1..N-1 = draft tokens, each with the index of its
parent.  Section 3.2 ("Single-pass token verification") verifies a chain;
a tree is the union of several retrieved chains, and a node may attend to
exactly the tokens that precede it on its own root path.
"""
import numpy as np


def validate(parent):
    """True iff ``parent`` is a topologically ordered tree rooted at 0."""
    parent = [int(p) for p in parent]
    if len(parent) == 0 or parent[0] != -1:
        return False
    return all(0 <= parent[j] < j for j in range(1, len(parent)))


def ancestors_or_self(parent, node):
    """Set of tree nodes on the path root -> node, both ends included."""
    out = set()
    u = int(node)
    while u >= 0:
        out.add(u)
        u = int(parent[u])
    return out


def depths(parent):
    """Depth of each node: number of edges between it and the root."""
    return np.array([len(ancestors_or_self(parent, n)) - 1 for n in range(len(parent))],
                    dtype=np.int64)


def ancestor_mask_bits(parent):
    """Per node, the sorted list of tree nodes it may attend to."""
    return [sorted(ancestors_or_self(parent, n)) for n in range(len(parent))]
