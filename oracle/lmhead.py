"""LM-head logits and greedy prediction, in float64.

Section 3.2: h_i is the decoder's final-layer state from which the model
predicts y_i, and verification compares each proposed token with the
model's greedy prediction.  The hidden states given here are taken after the
final norm; the head has no bias, no temperature and no soft-cap.

    logits[n, v] = sum_c hidden[n, c] * W[v, c]
    greedy[n]    = argmax_v logits[n, v]      (ties -> lowest v)
    margin[n]    = top-1 logit - top-2 logit  (flags near-ties)
"""
import numpy as np


def logits(hidden, weight, chunk=8192):
    """hidden [N, H], weight [V, H] -> float64 [N, V] (weight read in row chunks)."""
    hidden = np.asarray(hidden, dtype=np.float64)
    V = weight.shape[0]
    out = np.empty((hidden.shape[0], V), dtype=np.float64)
    for s in range(0, V, chunk):
        e = min(V, s + chunk)
        out[:, s:e] = hidden @ np.asarray(weight[s:e], dtype=np.float64).T
    return out


def greedy(lg):
    """Per row: (argmax with ties to the lowest index, top-2 margin, max)."""
    lg = np.asarray(lg, dtype=np.float64)
    am = np.argmax(lg, axis=1)                       # first maximal index
    top = lg[np.arange(lg.shape[0]), am]
    rest = lg.copy()
    rest[np.arange(lg.shape[0]), am] = -np.inf
    second = rest.max(axis=1) if lg.shape[1] > 1 else np.full(lg.shape[0], -np.inf)
    return am.astype(np.int64), top - second, top
