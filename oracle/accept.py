"""Acceptance of the proposal by greedy descent, Section 3.2.

The paper accepts the longest proposal prefix whose tokens equal the model's
greedy predictions, then appends the model's own prediction at the first
mismatch (or after the last draft), advancing the output by l_acc + 1
tokens.  On a tree the same rule descends from the root: at node u the
model predicts greedy[u]; if a child of u carries that token the walk moves
to it (the lowest-index such child if several do), otherwise it stops.

Returns (a, path, out_tokens, last):
  a          number of accepted draft tokens (l_acc)
  path       [a + 1] node indices, path[0] = root
  out_tokens [a + 1] accepted drafts followed by the model's bonus token
  last       path[a], the node whose state forms the next retrieval query
"""


def accept_walk(parent, tokens, greedy):
    n = len(parent)
    path = [0]
    while True:
        u = path[-1]
        want = int(greedy[u])
        nxt = None
        for c in range(n):
            if int(parent[c]) == u and int(tokens[c]) == want:
                nxt = c
                break
        if nxt is None:
            break
        path.append(nxt)
    a = len(path) - 1
    out_tokens = [int(tokens[c]) for c in path[1:]] + [int(greedy[path[-1]])]
    return a, path, out_tokens, path[-1]
