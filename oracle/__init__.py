"""fp64 CPU oracle of the verify step (test infrastructure only).

This package is the plain, slow, obviously correct statement of what the
verify step computes.  Only the tests, the smoke check and the benchmark's
CPU-baseline leg may import it; the CUDA library never uses it, and it never
imports the CUDA library.

Modules
  tree       ancestor sets and depths by walking parent indices
  attention  tree-masked GQA softmax attention over the reused prefix KV
  lmhead     LM-head logits, greedy argmax (ties -> lowest id), top-2 margin
  accept     greedy descent of the proposal tree (accepted length, tokens, path)
  commit     copy of the accepted path's K/V rows into the cache
  step       one whole verify step for one sequence, built from the above
  rope       rolling-image carryover: keys re-rotated to a new position
  retrieval  decoding-memory lookup: int8 query key, token-filtered cosine top-1

Every function is pinned by tests under ``tests/`` against brute force,
library special cases, closed forms and hand-derived fixtures.
"""
from . import tree, attention, lmhead, accept, commit, step, rope, retrieval  # noqa: F401
