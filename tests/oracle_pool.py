"""Oracle attention of many nodes in parallel, for the full-size parity tests.

Each worker regenerates one (workload, seed, layer, sequence) from the seeded
generator and runs oracle/attention.py on a subset of nodes.  Workers are
started with the "spawn" method and import numpy, the oracle and the input
generator only -- never torch or CUDA -- so the pool is safe beside a process
that already drives the GPU.
"""
from __future__ import annotations

import multiprocessing as mp
import os
from concurrent.futures import ProcessPoolExecutor

import numpy as np


def _values(x, dtype):
    from paper_2609_32166_gb300 import inputs as I
    return I.bf16_bits_to_f32(x) if dtype == "bf16" else np.asarray(x, dtype=np.float32)


def _oracle_nodes(job):
    """job = (workload, seed, layer, seq, nodes) -> [len(nodes), Hq, D] float64."""
    from oracle import attention as OA
    from paper_2609_32166_gb300 import inputs as I
    w, seed, layer, seq, nodes = job
    b = I.make_batch(w, seed)
    c0, c1 = int(b.cu_nodes[seq]), int(b.cu_nodes[seq + 1])
    q = _values(I.layer_q(w, b, layer), w.dtype)[c0:c1]
    tk, tv = (_values(x, w.dtype)[c0:c1] for x in I.layer_tree_kv(w, b, layer))
    pk, pv = (_values(x, w.dtype) for x in I.layer_prefix_kv(w, b, layer, seq))
    out = OA.tree_attention(q, pk, pv, tk, tv, b.parents[seq], nodes=nodes)
    return out[list(nodes)]


def make_pool(workers: int = None) -> ProcessPoolExecutor:
    n = workers or max(1, min(16, (os.cpu_count() or 2) - 1))
    return ProcessPoolExecutor(max_workers=n, mp_context=mp.get_context("spawn"))


def oracle_attention_nodes(pool, w, seed, layer, seq, nodes, chunk: int = 4) -> dict:
    """{node: [Hq, D] float64} for every node in `nodes`, computed in chunks."""
    nodes = list(nodes)
    jobs = [(w, seed, layer, seq, nodes[i:i + chunk]) for i in range(0, len(nodes), chunk)]
    out = {}
    for job, res in zip(jobs, pool.map(_oracle_nodes, jobs)):
        for n, r in zip(job[4], res):
            out[n] = r
    return out
