"""The seeded input generator: determinism, shapes and tree constraints."""
import os
import re

import numpy as np
import pytest

from paper_2609_32166_gb300 import inputs as I
from oracle import tree as T

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3, 1.0 + 2**-8 + 2**-12], np.float32)
    bits = I.round_to_bf16_bits(x)
    back = I.bf16_bits_to_f32(bits)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: even mantissa wins (1.0)
    assert back[1] == 1.0
    # 1 + 3*2^-8 is a tie between 1+2^-7 and 1+2^-6: even wins (1 + 2^-6)
    assert back[2] == np.float32(1.0 + 2**-6)
    assert back[5] == np.float32(1.0 + 2**-7)
    assert back[0] == 1.0 and back[3] == -2.5
    assert abs(back[4] - 3.0e-3) <= 3.0e-3 * 2**-8


def test_streams_are_deterministic_and_independent():
    a = I.normal((64, 8), 1.0, 0, "q", 3, "bf16")
    b = I.normal((64, 8), 1.0, 0, "q", 3, "bf16")
    c = I.normal((64, 8), 1.0, 0, "q", 4, "bf16")
    assert a.dtype == np.uint16 and np.array_equal(a, b) and not np.array_equal(a, c)
    f = I.normal((1000,), 0.02, 1, "w", 0, "f32")
    assert f.dtype == np.float32 and 0.015 < f.std() < 0.025


@pytest.mark.parametrize("name", sorted(I.WORKLOADS))
def test_workload_structure(name):
    w = I.WORKLOADS[name]
    b = I.make_batch(w, seed=0)
    assert len(b.parents) == w.batch
    for s, p in enumerate(b.parents):
        assert len(p) == w.nodes and T.validate(p)
        assert T.depths(p).max() <= w.max_depth
        if w.tree == "random":
            assert max(np.bincount(p[1:], minlength=w.nodes)) <= w.branching
        assert 0 <= b.forced_end[s] < w.nodes
        assert w.prefix[0] <= b.prefix_lens[s] <= w.prefix[1]
    if w.layout == "paged":
        assert sorted(b.page_table.ravel()) == list(range(b.num_pages))
        need = -(-(int(b.prefix_lens.max()) + w.nodes) // I.PAGE_SIZE)
        assert b.page_table.shape[1] >= need


def test_planted_tokens_fix_the_accepted_path():
    w = I.WORKLOADS["7b-bf16-batch8-paged"]
    b = I.make_batch(w, seed=3)
    rng = np.random.default_rng(0)
    argmax = rng.integers(0, w.vocab, size=b.total_nodes)
    tok = I.plant_tokens(b, argmax)
    cu = b.cu_nodes
    from oracle.accept import accept_walk
    for s, p in enumerate(b.parents):
        t = tok[cu[s]:cu[s + 1]]
        g = argmax[cu[s]:cu[s + 1]]
        a, path, _, last = accept_walk(p, t, g)
        assert path == I.root_path(p, int(b.forced_end[s]))


def test_chains_tree_has_requested_shape():
    rng = np.random.default_rng(0)
    p = I.chains_tree(128, 24, rng)
    assert len(p) == 128 and T.depths(p).max() == 24


def test_paged_placement_round_trip():
    w = I.scaled(I.WORKLOADS["7b-bf16-batch8-paged"], hq=4, hkv=2, d=16, prefix=(20, 50), nodes=5)
    b = I.make_batch(w, seed=1)
    cache = np.zeros(I.cache_shape(w, b), dtype=np.uint16)
    rows = []
    for s in range(w.batch):
        r = I.layer_prefix_kv(w, b, 0, s)[0]
        I.place_prefix(w, b, cache, s, r)
        rows.append(r)
    for s in range(w.batch):
        assert np.array_equal(I.cache_rows(w, b, cache, s, 0, int(b.prefix_lens[s])), rows[s])


def test_oracle_and_library_are_independent():
    """The oracle never imports the package and the package never imports the oracle."""
    for d, banned in (("oracle", r"paper_2609_32166_gb300"),
                      ("paper_2609_32166_gb300", r"\boracle\b")):
        for root, _, files in os.walk(os.path.join(ROOT, d)):
            for f in files:
                if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp", ".c")):
                    src = open(os.path.join(root, f)).read()
                    imports = [l for l in src.splitlines() if re.match(r"\s*(import|from|#include)\b", l)]
                    assert not any(re.search(banned, l) for l in imports), (f, imports)
