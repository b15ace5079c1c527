"""Seeded synthetic inputs for the verify step (shared by tests, bench and smoke).

This module draws random numbers and lays them out; it holds none of the
verification arithmetic (no attention, no logits, no acceptance).  Both the
CUDA path and the fp64 oracle receive exactly the arrays produced here.

Shapes follow the five workloads named in ``WORKLOADS``: a tiny fp32 chain,
a 2B-VLM-shaped chain, a 7B-VLM-shaped 64-node tree, an 8-sequence paged
batch and a 32K-token long-context tree.  Values are N(0, 1) for Q, K, V and
hidden states and N(0, 0.02) for the LM-head weight, rounded to bf16
(round-to-nearest-even) for the bf16 workloads.

Every tensor has its own counter-keyed stream (seed, tensor tag, index), so
any single layer can be regenerated without drawing the others.

The proposal's draft tokens depend on the model's greedy predictions
(Section 3.2: a draft is accepted only where it equals the greedy token), so
tree *structure* and the forced accepted path are drawn here, and
``plant_tokens`` fills the draft tokens once a caller supplies the argmax of
each node.
"""
from __future__ import annotations

import dataclasses
import zlib
from typing import List, Optional

import numpy as np

PAGE_SIZE = 16
MAX_NODES = 128


# ----------------------------------------------------------------------------
# random streams and bf16 rounding
# ----------------------------------------------------------------------------
def _stream(seed: int, tag: str, index: int = 0) -> np.random.Generator:
    key = (zlib.crc32(tag.encode()), int(index))
    ss = np.random.SeedSequence(entropy=int(seed), spawn_key=key)
    return np.random.Generator(np.random.Philox(ss))


def round_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit patterns (uint16), round to nearest, ties to even."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> np.uint32(16)) & np.uint32(1)
    r = (u + np.uint32(0x7FFF) + lsb) >> np.uint32(16)
    return r.astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


def normal(shape, std: float, seed: int, tag: str, index: int, dtype: str,
           chunk: int = 1 << 24) -> np.ndarray:
    """N(0, std^2) samples of ``shape``: float32 for dtype 'f32', bf16 bit
    patterns (uint16) for dtype 'bf16'.  Drawn in chunks to bound host memory."""
    rng = _stream(seed, tag, index)
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.float32 if dtype == "f32" else np.uint16)
    for s in range(0, n, chunk):
        e = min(n, s + chunk)
        x = rng.standard_normal(e - s, dtype=np.float32)
        if std != 1.0:
            x *= np.float32(std)
        out[s:e] = x if dtype == "f32" else round_to_bf16_bits(x)
    return out.reshape(shape)


def as_f64(x: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 view of generated values (bf16 bits or float32)."""
    if dtype == "bf16":
        return bf16_bits_to_f32(x).astype(np.float64)
    return x.astype(np.float64)


# ----------------------------------------------------------------------------
# workloads
# ----------------------------------------------------------------------------
@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    dtype: str            # "f32" | "bf16"
    layers: int
    batch: int
    hq: int
    hkv: int
    d: int
    hidden: int
    vocab: int
    prefix: tuple         # (lo, hi) inclusive range of prefix lengths
    nodes: int            # tree nodes per sequence, root included
    tree: str             # "chain" | "chains" | "random"
    max_depth: int
    accept: str           # "chain" | "uniform_node" | "uniform_depth"
    layout: str           # "contiguous" | "paged"
    branching: int = 3

    @property
    def group(self) -> int:
        return self.hq // self.hkv


WORKLOADS = {
    "tiny-f32-chain8": Workload(
        "tiny-f32-chain8", "f32", 1, 1, 4, 1, 64, 256, 1024, (256, 256), 9,
        "chain", 8, "chain", "contiguous"),
    "2b-bf16-chain16": Workload(
        "2b-bf16-chain16", "bf16", 28, 1, 12, 2, 128, 1536, 151936,
        (1800, 1800), 17, "chain", 16, "chain", "contiguous"),
    "7b-bf16-tree64": Workload(
        "7b-bf16-tree64", "bf16", 28, 1, 28, 4, 128, 3584, 152064,
        (4096, 4096), 64, "chains", 12, "uniform_node", "contiguous"),
    "7b-bf16-batch8-paged": Workload(
        "7b-bf16-batch8-paged", "bf16", 28, 8, 28, 4, 128, 3584, 152064,
        (2048, 6144), 32, "random", 31, "uniform_node", "paged"),
    "7b-bf16-32k-tree128": Workload(
        "7b-bf16-32k-tree128", "bf16", 28, 1, 28, 4, 128, 3584, 152064,
        (32768, 32768), 128, "chains", 24, "uniform_depth", "contiguous"),
}


def scaled(w: Workload, **kw) -> Workload:
    """A copy of ``w`` with some fields replaced (small parity cases)."""
    return dataclasses.replace(w, **kw)


# ----------------------------------------------------------------------------
# proposal trees
# ----------------------------------------------------------------------------
def chain_tree(n: int) -> np.ndarray:
    return np.arange(-1, n - 1, dtype=np.int32)


def chains_tree(n: int, max_depth: int, rng: np.random.Generator) -> np.ndarray:
    """Union of retrieved candidate chains sharing prefixes: the first chain
    runs from the root to ``max_depth``; each later chain branches off a
    random node of the tree built so far and runs down to ``max_depth``
    (the last one truncated so the tree has exactly ``n`` nodes)."""
    parent = [-1]
    depth = [0]
    first = True
    while len(parent) < n:
        if first:
            u = 0
            first = False
        else:
            cand = [i for i in range(len(parent)) if depth[i] < max_depth]
            u = int(cand[rng.integers(len(cand))])
        while depth[u] < max_depth and len(parent) < n:
            parent.append(u)
            depth.append(depth[u] + 1)
            u = len(parent) - 1
    return np.asarray(parent, dtype=np.int32)


def random_tree(n: int, branching: int, rng: np.random.Generator) -> np.ndarray:
    """Random recursive tree: each new node picks a parent uniformly among
    the nodes that still have fewer than ``branching`` children."""
    parent = [-1]
    nchild = [0]
    for _ in range(1, n):
        cand = [i for i in range(len(parent)) if nchild[i] < branching]
        u = int(cand[rng.integers(len(cand))])
        parent.append(u)
        nchild[u] += 1
        nchild.append(0)
    return np.asarray(parent, dtype=np.int32)


def node_depths(parent: np.ndarray) -> np.ndarray:
    d = np.zeros(len(parent), dtype=np.int32)
    for j in range(1, len(parent)):
        d[j] = d[parent[j]] + 1
    return d


def root_path(parent: np.ndarray, node: int) -> List[int]:
    p = [int(node)]
    while parent[p[-1]] >= 0:
        p.append(int(parent[p[-1]]))
    return p[::-1]


@dataclasses.dataclass
class Batch:
    """Structure of one verify step: trees, prefix lengths, forced paths."""
    workload: Workload
    seed: int
    parents: List[np.ndarray]      # per sequence, local indices, parent[0] = -1
    prefix_lens: np.ndarray        # [B] int32
    forced_end: np.ndarray         # [B] node where the planted accepted path ends
    page_table: Optional[np.ndarray]  # [B, pages_per_seq] int32 (paged only)
    num_pages: int
    max_seq: int                   # contiguous: rows per (sequence, head)

    @property
    def cu_nodes(self) -> np.ndarray:
        c = np.zeros(len(self.parents) + 1, dtype=np.int32)
        c[1:] = np.cumsum([len(p) for p in self.parents])
        return c

    @property
    def total_nodes(self) -> int:
        return int(sum(len(p) for p in self.parents))

    @property
    def parent_flat(self) -> np.ndarray:
        return np.concatenate(self.parents).astype(np.int32)


def _draw_end(w: Workload, parent: np.ndarray, rng: np.random.Generator) -> int:
    """End node of the planted accepted path, by the workload's rule."""
    if w.accept in ("chain", "uniform_node"):
        return int(rng.integers(0, len(parent)))       # chain: a ~ U[0, nodes-1]
    dep = node_depths(parent)
    a = int(rng.integers(0, int(dep.max()) + 1))
    cand = np.nonzero(dep == a)[0]
    return int(cand[rng.integers(len(cand))])


def step_forced_ends(batch: "Batch", count: int) -> List[np.ndarray]:
    """Planted accepted-path ends for ``count`` successive verify steps over
    the same trees (each step verifies a new proposal)."""
    rng = _stream(batch.seed, "step_ends")
    return [np.asarray([_draw_end(batch.workload, p, rng) for p in batch.parents], np.int32)
            for _ in range(count)]


def make_batch(w: Workload, seed: int = 0) -> Batch:
    rng = _stream(seed, "structure")
    parents, ends = [], []
    lo, hi = w.prefix
    prefix_lens = rng.integers(lo, hi + 1, size=w.batch).astype(np.int32)
    for b in range(w.batch):
        if w.tree == "chain":
            p = chain_tree(w.nodes)
        elif w.tree == "chains":
            p = chains_tree(w.nodes, w.max_depth, rng)
        else:
            p = random_tree(w.nodes, w.branching, rng)
        end = _draw_end(w, p, rng)
        parents.append(p)
        ends.append(end)
    max_seq = int(prefix_lens.max()) + w.nodes
    page_table, num_pages = None, 0
    if w.layout == "paged":
        per_seq = -(-max_seq // PAGE_SIZE)
        num_pages = per_seq * w.batch
        perm = rng.permutation(num_pages).astype(np.int32)
        page_table = perm.reshape(w.batch, per_seq)
    return Batch(w, seed, parents, prefix_lens, np.asarray(ends, np.int32),
                 page_table, num_pages, max_seq)


def plant_tokens(batch: Batch, argmax: np.ndarray, forced_end=None, salt: int = 0) -> np.ndarray:
    """Draft tokens for every node given each node's greedy token ``argmax``
    (flat over the batch).  Along the planted path the child's token is its
    parent's greedy token; every other child gets a token different from its
    parent's greedy token and from its siblings', so the accepted path is
    exactly the planted one.  The root's token (the current token) is random."""
    w = batch.workload
    rng = _stream(batch.seed, "tokens", salt)
    ends = batch.forced_end if forced_end is None else forced_end
    out = np.empty(batch.total_nodes, dtype=np.int32)
    cu = batch.cu_nodes
    for b, parent in enumerate(batch.parents):
        off = int(cu[b])
        on_path = set(root_path(parent, int(ends[b])))
        used = {}
        out[off] = int(rng.integers(0, w.vocab))
        for j in range(1, len(parent)):
            u = int(parent[j])
            g = int(argmax[off + u])
            sib = used.setdefault(u, set())
            if j in on_path:
                t = g
            else:
                while True:
                    t = int(rng.integers(0, w.vocab - 1))
                    t = t + 1 if t >= g else t
                    if t not in sib:
                        break
            sib.add(t)
            out[off + j] = t
    return out


# ----------------------------------------------------------------------------
# per-layer tensors and cache placement
# ----------------------------------------------------------------------------
def layer_q(w: Workload, batch: Batch, layer: int) -> np.ndarray:
    return normal((batch.total_nodes, w.hq, w.d), 1.0, batch.seed, "q", layer, w.dtype)


def layer_tree_kv(w: Workload, batch: Batch, layer: int):
    shp = (batch.total_nodes, w.hkv, w.d)
    return (normal(shp, 1.0, batch.seed, "tree_k", layer, w.dtype),
            normal(shp, 1.0, batch.seed, "tree_v", layer, w.dtype))


def layer_prefix_kv(w: Workload, batch: Batch, layer: int, seq: int):
    """Prefix K, V of one sequence and layer: [Hkv, P_b, D] each."""
    shp = (w.hkv, int(batch.prefix_lens[seq]), w.d)
    idx = layer * 4096 + seq
    return (normal(shp, 1.0, batch.seed, "prefix_k", idx, w.dtype),
            normal(shp, 1.0, batch.seed, "prefix_v", idx, w.dtype))


def hidden_states(w: Workload, batch: Batch) -> np.ndarray:
    return normal((batch.total_nodes, w.hidden), 1.0, batch.seed, "hidden", 0, w.dtype)


def lm_weight(w: Workload, seed: int) -> np.ndarray:
    return normal((w.vocab, w.hidden), 0.02, seed, "lm_weight", 0, w.dtype)


def cache_shape(w: Workload, batch: Batch):
    """Shape of one layer's K (or V) cache in the workload's layout."""
    if w.layout == "paged":
        return (batch.num_pages, w.hkv, PAGE_SIZE, w.d)
    return (w.batch, w.hkv, batch.max_seq, w.d)


def place_prefix(w: Workload, batch: Batch, cache: np.ndarray, seq: int,
                 rows: np.ndarray) -> None:
    """Write a sequence's prefix rows [Hkv, P, D] at positions 0..P-1 of one
    layer's cache (contiguous [B, Hkv, S, D] or paged [pages, Hkv, 16, D])."""
    P = rows.shape[1]
    if w.layout == "contiguous":
        cache[seq, :, :P, :] = rows
        return
    pt = batch.page_table[seq]
    for p0 in range(0, P, PAGE_SIZE):
        n = min(PAGE_SIZE, P - p0)
        cache[pt[p0 // PAGE_SIZE], :, :n, :] = rows[:, p0:p0 + n, :]


def cache_rows(w: Workload, batch: Batch, cache: np.ndarray, seq: int,
               start: int, count: int) -> np.ndarray:
    """Read positions start..start+count-1 of one sequence: [Hkv, count, D]."""
    if w.layout == "contiguous":
        return cache[seq, :, start:start + count, :]
    out = np.empty((w.hkv, count, w.d), dtype=cache.dtype)
    pt = batch.page_table[seq]
    for i in range(count):
        pos = start + i
        out[:, i, :] = cache[pt[pos // PAGE_SIZE], :, pos % PAGE_SIZE, :]
    return out


# ----------------------------------------------------------------------------
# rolling-image carryover and decoding-memory inputs
# ----------------------------------------------------------------------------
KEY_DIM = 256
QWEN_VOCAB = 151936


def page_table(n_seqs: int, pages_per_seq: int, seed: int, spare: int = 3):
    """A random permutation of n_seqs * pages_per_seq + spare pages laid out
    as page_table [n_seqs, pages_per_seq]; returns (table int32, num_pages)."""
    num_pages = n_seqs * pages_per_seq + spare
    perm = _stream(seed, "page_table").permutation(num_pages).astype(np.int32)
    return perm[: n_seqs * pages_per_seq].reshape(n_seqs, pages_per_seq), num_pages


def int8_keys(n: int, seed: int, tag: str = "memory_keys", index: int = 0) -> np.ndarray:
    """[n, 256] int8: N(0, 40^2) rounded and clipped to [-127, 127] (the spread
    of keys that use most of the int8 range)."""
    rng = _stream(seed, tag, index)
    x = rng.normal(0.0, 40.0, size=(n, KEY_DIM))
    return np.clip(np.rint(x), -127, 127).astype(np.int8)


@dataclasses.dataclass
class Memory:
    keys: np.ndarray    # [M, 256] int8
    token: np.ndarray   # [M] int32, token of the shared array at the entry's position
    pos: np.ndarray     # [M] int32, position of the entry in the shared token array
    bound: np.ndarray   # [M] int32, last position of the entry's output sequence


def decoding_memory(n_entries: int, seed: int, vocab: int = QWEN_VOCAB,
                    mean_len: int = 80) -> Memory:
    """A decoding-experience memory of n_entries: output sequences of
    U[16, 2 * mean_len - 16] tokens appended to one shared token array, one
    entry per position (the last position of each sequence is its boundary).
    Tokens follow a Zipf(1.2) law over the vocabulary, so a query's token
    matches anywhere from a handful to a few percent of the entries."""
    rng = _stream(seed, "memory_layout")
    bound = np.empty(n_entries, dtype=np.int32)
    p = 0
    while p < n_entries:
        n = int(rng.integers(16, max(17, 2 * mean_len - 15)))
        e = min(n_entries, p + n)
        bound[p:e] = p + n - 1
        p = e
    token = ((rng.zipf(1.2, size=n_entries) - 1) % vocab).astype(np.int32)
    pos = np.arange(n_entries, dtype=np.int32)
    return Memory(int8_keys(n_entries, seed), token, pos, bound)
