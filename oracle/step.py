"""One whole verify step for one sequence (Section 3.2), in float64.

Attention of every layer over the reused prefix, then LM head, greedy
prediction and acceptance, then the commit of the accepted rows.  The
per-layer queries and tree K/V are inputs: the projections and MLPs that
produce them are outside the verify path.
"""
from .attention import tree_attention
from .lmhead import logits, greedy
from .accept import accept_walk
from .commit import commit_rows


def verify_step(layers, hidden, weight, parent, tokens, prefix_len):
    """layers: list of dicts with q, prefix_k, prefix_v, tree_k, tree_v and
    cache_k, cache_v ([Hkv, S, D] rows of this sequence).  Returns a dict."""
    outs = [tree_attention(L["q"], L["prefix_k"], L["prefix_v"], L["tree_k"],
                           L["tree_v"], parent) for L in layers]
    lg = logits(hidden, weight)
    am, margin, top = greedy(lg)
    a, path, out_tokens, last = accept_walk(parent, tokens, am)
    caches = []
    for L in layers:
        ck, n1 = commit_rows(L["cache_k"], prefix_len, path, L["tree_k"])
        cv, _ = commit_rows(L["cache_v"], prefix_len, path, L["tree_v"])
        caches.append((ck, cv))
    return dict(attn=outs, argmax=am, margin=margin, max_logit=top, accept_len=a,
                path=path, out_tokens=out_tokens, last_node=last, caches=caches,
                new_len=n1)
