"""The C-ABI library on the CPU: it loads, exports every declared symbol,
builds ancestor bitmaps that agree with the oracle's parent walk, and
rejects bad arguments with a status code before touching a GPU."""
import ctypes as C

import numpy as np
import pytest

from oracle import tree as OT
from paper_2609_32166_gb300 import _build
from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I


@pytest.fixture(scope="module", autouse=True)
def built():
    _build.build()


def test_exports_every_declared_symbol():
    names = pb.header_functions()
    assert set(names) >= {"pf_tree_prepare", "pf_verify_attention", "pf_lmhead_accept",
                          "pf_lmhead_accept_workspace_size", "pf_kv_commit", "pf_last_error",
                          "pf_version"}
    L = pb.lib()
    for n in names:
        assert hasattr(L, n), n
    assert pb.pf_version() >= 100


def test_struct_layouts_match_header():
    """ctypes mirrors match the C structs (sizes from a compiled probe)."""
    import os
    import subprocess
    import tempfile
    src = r'''
#include <stdio.h>
#include <stddef.h>
#include "pf_verify.h"
int main(void) {
  printf("%zu %zu %zu %zu %zu %zu %zu\n", sizeof(pf_kv_view), sizeof(pf_attn_desc),
         sizeof(pf_lm_desc), sizeof(pf_commit_desc), offsetof(pf_attn_desc, cache),
         offsetof(pf_commit_desc, cache), offsetof(pf_commit_desc, new_len));
  return 0;
}
'''
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "probe.c")
        exe = os.path.join(d, "probe")
        open(c, "w").write(src)
        subprocess.run(["gcc", "-I", _build.INCLUDE, c, "-o", exe], check=True)
        got = [int(x) for x in subprocess.run([exe], capture_output=True, text=True,
                                              check=True).stdout.split()]
    want = [C.sizeof(pb.pf_kv_view), C.sizeof(pb.pf_attn_desc), C.sizeof(pb.pf_lm_desc),
            C.sizeof(pb.pf_commit_desc), pb.pf_attn_desc.cache.offset,
            pb.pf_commit_desc.cache.offset, pb.pf_commit_desc.new_len.offset]
    assert got == want


@pytest.mark.parametrize("name", sorted(I.WORKLOADS))
def test_tree_prepare_matches_parent_walk(name):
    w = I.WORKLOADS[name]
    b = I.make_batch(w, seed=2)
    for parent in b.parents:
        depth, mask = pb.pf_tree_prepare(parent)
        assert list(depth) == list(OT.depths(parent))
        for j in range(len(parent)):
            bits = {i for i in range(len(parent)) if (int(mask[j, i >> 6]) >> (i & 63)) & 1}
            assert bits == OT.ancestors_or_self(parent, j)


def test_tree_prepare_max_and_rejects():
    rng = np.random.default_rng(0)
    p = I.random_tree(128, 5, rng)
    depth, mask = pb.pf_tree_prepare(p)
    assert mask.shape == (128, 2)
    for bad, status in (([0], pb.PF_ERR_TREE), ([-1, 1], pb.PF_ERR_TREE),
                        ([-1, 0, 2], pb.PF_ERR_TREE), ([-1, -1], pb.PF_ERR_TREE),
                        (list(range(-1, 128)), pb.PF_ERR_SHAPE)):
        with pytest.raises(pb.PfError) as e:
            pb.pf_tree_prepare(bad)
        assert e.value.status == status
    with pytest.raises(pb.PfError) as e:
        pb.pf_tree_prepare([])
    assert e.value.status == pb.PF_ERR_SHAPE


def _attn_desc(**kw):
    d = pb.pf_attn_desc()
    d.dtype, d.batch, d.n_q_heads, d.n_kv_heads, d.head_dim = pb.PF_BF16, 1, 4, 2, 128
    d.total_nodes, d.max_nodes, d.max_prefix_len = 3, 3, 10
    fake = 0x10000
    for f in ("cu_nodes", "prefix_len", "q", "tree_k", "tree_v", "mask", "out"):
        setattr(d, f, fake)
    d.cache.layout, d.cache.k, d.cache.v, d.cache.max_seq = pb.PF_KV_CONTIGUOUS, fake, fake, 64
    for k, v in kw.items():
        if k.startswith("cache_"):
            setattr(d.cache, k[6:], v)
        else:
            setattr(d, k, v)
    return d


@pytest.mark.parametrize("kw,status", [
    (dict(q=None), pb.PF_ERR_NULL),
    (dict(dtype=7), pb.PF_ERR_DTYPE),
    (dict(n_q_heads=5), pb.PF_ERR_SHAPE),
    (dict(head_dim=96), pb.PF_ERR_SHAPE),
    (dict(max_nodes=129), pb.PF_ERR_SHAPE),
    (dict(max_nodes=0), pb.PF_ERR_SHAPE),
    (dict(max_prefix_len=65), pb.PF_ERR_CAPACITY),
    (dict(cache_layout=1, cache_page_table=None), pb.PF_ERR_NULL),
    (dict(cache_layout=1, cache_page_table=0x10000, cache_num_pages=4, cache_pages_per_seq=0),
     pb.PF_ERR_SHAPE),
    (dict(cache_layout=1, cache_page_table=0x10000, cache_num_pages=4, cache_pages_per_seq=1,
          max_prefix_len=17), pb.PF_ERR_CAPACITY),
    (dict(q=0x10008), pb.PF_ERR_ALIGN),
])
def test_attention_rejects_bad_arguments(kw, status):
    with pytest.raises(pb.PfError) as e:
        pb.pf_verify_attention(_attn_desc(**kw), 0)
    assert e.value.status == status
    assert pb.pf_last_error()


def _lm_desc(**kw):
    d = pb.pf_lm_desc()
    d.dtype, d.batch, d.hidden, d.vocab = pb.PF_BF16, 1, 64, 1000
    d.total_nodes, d.max_nodes = 4, 4
    fake = 0x10000
    for f in ("cu_nodes", "hidden_states", "weight", "tokens", "parent", "argmax",
              "accept_len", "path", "out_tokens"):
        setattr(d, f, fake)
    for k, v in kw.items():
        setattr(d, k, v)
    return d


@pytest.mark.parametrize("kw,ws,status", [
    (dict(weight=None), 4096, pb.PF_ERR_NULL),
    (dict(), 16, pb.PF_ERR_WORKSPACE),
    (dict(total_nodes=257), 4096, pb.PF_ERR_SHAPE),
    (dict(total_nodes=0), 4096, pb.PF_ERR_SHAPE),
    (dict(hidden=100), 4096, pb.PF_ERR_ALIGN),
    (dict(dtype=2), 4096, pb.PF_ERR_DTYPE),
    (dict(max_nodes=200), 4096, pb.PF_ERR_SHAPE),
])
def test_lmhead_rejects_bad_arguments(kw, ws, status):
    with pytest.raises(pb.PfError) as e:
        pb.pf_lmhead_accept(_lm_desc(**kw), 0x20000, ws, 0)
    assert e.value.status == status


def _commit_desc(**kw):
    d = pb.pf_commit_desc()
    d.dtype, d.batch, d.n_layers, d.n_kv_heads, d.head_dim = pb.PF_BF16, 1, 2, 2, 128
    d.total_nodes, d.max_nodes, d.max_prefix_len = 5, 5, 20
    fake = 0x10000
    for f in ("cu_nodes", "prefix_len", "accept_len", "path", "tree_k", "tree_v"):
        setattr(d, f, fake)
    d.new_len = 0x30000
    d.tree_layer_stride, d.cache_layer_stride = 5 * 2 * 128, 2 * 64 * 128
    d.cache.layout, d.cache.k, d.cache.v, d.cache.max_seq = pb.PF_KV_CONTIGUOUS, fake, fake, 64
    for k, v in kw.items():
        if k.startswith("cache_"):
            setattr(d.cache, k[6:], v)
        else:
            setattr(d, k, v)
    return d


@pytest.mark.parametrize("kw,status", [
    (dict(path=None), pb.PF_ERR_NULL),
    (dict(new_len=0x10000), pb.PF_ERR_SHAPE),
    (dict(cache_max_seq=24), pb.PF_ERR_CAPACITY),
    (dict(head_dim=4), pb.PF_ERR_ALIGN),
    (dict(tree_layer_stride=3), pb.PF_ERR_ALIGN),
    (dict(n_layers=0), pb.PF_ERR_SHAPE),
    (dict(cache_layout=1, cache_page_table=0x10000, cache_num_pages=3, cache_pages_per_seq=1),
     pb.PF_ERR_CAPACITY),
])
def test_commit_rejects_bad_arguments(kw, status):
    with pytest.raises(pb.PfError) as e:
        pb.pf_kv_commit(_commit_desc(**kw), 0)
    assert e.value.status == status
