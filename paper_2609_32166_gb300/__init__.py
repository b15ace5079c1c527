"""GB300-native verify step of retrieval-based multi-token proposals.

The hot path (tree-masked attention over a reused KV cache, LM head with
greedy acceptance, and commit of the accepted K/V rows) lives in the CUDA
library ``libpfverify.so`` built from ``csrc/``; ``binding`` marshals
arguments to its C ABI.  ``inputs`` draws the seeded synthetic workloads.
"""
