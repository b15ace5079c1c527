"""Prompt-prefix KV carryover: the longest identical prefix of two prompts.

Section 3.4 ("Prompt-prefix KV-state carryover"): consecutive action-step
prompts P_t and P_{t+1} of one task share a prefix of identical tokens;
with p the length of their longest identical prefix, the cached K/V of
positions 0 .. p-1 stay valid (same content, positions and causal context)
and computation resumes at position p.

Reading (the paper is silent on the representation): a prompt is a
sequence of integer token keys in which text tokens are their token ids and
image tokens carry an identifier of the image content at that position, so
that "identical" covers both the token and what it shows.  Cached rows at
positions >= p are stale; the cache length becomes p.

Test infrastructure only: imported by tests, never by the library.
"""


def common_prefix(prev, nxt):
    """Length p of the longest common prefix of two key sequences."""
    p = 0
    n = min(len(prev), len(nxt))
    while p < n and int(prev[p]) == int(nxt[p]):
        p += 1
    return p


def carry_over(prev, nxt):
    """(p, new cache length, positions to compute for the new prompt)."""
    p = common_prefix(prev, nxt)
    return p, p, len(nxt) - p
