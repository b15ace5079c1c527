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
                          "pf_version", "pf_kv_shift", "pf_retrieval_key", "pf_retrieve",
                          "pf_retrieval_workspace_size", "pf_lmhead_accept_noalloc",
                          "pf_prefix_match", "pf_selftest_wait", "pf_controller_init",
                          "pf_controller_observe", "pf_controller_choose", "pf_length_select"}
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
  printf("%zu %zu %zu %zu %zu %zu %zu\n", sizeof(pf_shift_desc), offsetof(pf_shift_desc, cache),
         offsetof(pf_shift_desc, cache_layer_stride), sizeof(pf_key_desc),
         offsetof(pf_key_desc, key_out), sizeof(pf_retrieval_desc),
         offsetof(pf_retrieval_desc, similarity));
  printf("%zu %zu\n", sizeof(pf_prefix_desc), offsetof(pf_prefix_desc, cache_len));
  printf("%zu %zu\n", offsetof(pf_attn_desc, workspace), offsetof(pf_attn_desc, workspace_bytes));
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
            pb.pf_commit_desc.cache.offset, pb.pf_commit_desc.new_len.offset,
            C.sizeof(pb.pf_shift_desc), pb.pf_shift_desc.cache.offset,
            pb.pf_shift_desc.cache_layer_stride.offset, C.sizeof(pb.pf_key_desc),
            pb.pf_key_desc.key_out.offset, C.sizeof(pb.pf_retrieval_desc),
            pb.pf_retrieval_desc.similarity.offset,
            C.sizeof(pb.pf_prefix_desc), pb.pf_prefix_desc.cache_len.offset,
            pb.pf_attn_desc.workspace.offset, pb.pf_attn_desc.workspace_bytes.offset]
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
    # launch fields
    (dict(kernel=8), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TWO_BLOCK, head_dim=64), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TWO_BLOCK, stages=3), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TWO_BLOCK, rows_per_cta=256), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TWO_BLOCK, splits=17), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_STREAM, splits=2), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_BATCH, splits=2), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_BATCH, head_dim=64), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_BATCH, stages=2), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_BATCH, rows_per_cta=128), pb.PF_ERR_SHAPE),
    (dict(kernel=-1), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_PAIR, splits=9), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TC64, splits=17), pb.PF_ERR_SHAPE),
    (dict(splits=-1), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_PAIR, head_dim=64), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TC128, rows_per_cta=128), pb.PF_ERR_SHAPE),
    (dict(rows_per_cta=192), pb.PF_ERR_SHAPE),
    (dict(rows_per_cta=128, n_q_heads=258, n_kv_heads=2), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TC64, stages=2), pb.PF_ERR_SHAPE),
    (dict(kernel=pb.PF_ATTN_KERNEL_TC128, stages=4), pb.PF_ERR_SHAPE),
    (dict(dtype=pb.PF_F32, kernel=pb.PF_ATTN_KERNEL_MMA), pb.PF_ERR_DTYPE),
    (dict(dtype=pb.PF_F32, splits=2), pb.PF_ERR_DTYPE),
    (dict(flags=8), pb.PF_ERR_SHAPE),
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


def _shift_desc(**kw):
    d = pb.pf_shift_desc()
    d.dtype, d.n_layers, d.n_kv_heads, d.head_dim = pb.PF_BF16, 2, 2, 128
    d.seq, d.batch, d.src, d.dst, d.count, d.rope_base = 0, 1, 10, 4, 20, 1e4
    fake = 0x10000
    d.cache_layer_stride = 2 * 64 * 128
    d.cache.layout, d.cache.k, d.cache.v, d.cache.max_seq = pb.PF_KV_CONTIGUOUS, fake, fake, 64
    for k, v in kw.items():
        if k.startswith("cache_") and k != "cache_layer_stride":
            setattr(d.cache, k[6:], v)
        else:
            setattr(d, k, v)
    return d


@pytest.mark.parametrize("kw,status", [
    (dict(cache_k=None), pb.PF_ERR_NULL),
    (dict(dtype=5), pb.PF_ERR_DTYPE),
    (dict(head_dim=130), pb.PF_ERR_SHAPE),
    (dict(head_dim=8), pb.PF_ERR_SHAPE),          # half a bf16 row below 16 bytes
    (dict(head_dim=512), pb.PF_ERR_SHAPE),
    (dict(count=-1), pb.PF_ERR_SHAPE),
    (dict(src=-3), pb.PF_ERR_SHAPE),
    (dict(rope_base=0.0), pb.PF_ERR_SHAPE),
    (dict(seq=1), pb.PF_ERR_SHAPE),
    (dict(n_layers=0), pb.PF_ERR_SHAPE),
    (dict(dst=50), pb.PF_ERR_CAPACITY),           # 50 + 20 rows > max_seq 64
    (dict(cache_layout=1, cache_page_table=0x10000, cache_num_pages=8, cache_pages_per_seq=1),
     pb.PF_ERR_CAPACITY),
    (dict(cache_layer_stride=3), pb.PF_ERR_ALIGN),
])
def test_kv_shift_rejects_bad_arguments(kw, status):
    with pytest.raises(pb.PfError) as e:
        pb.pf_kv_shift(_shift_desc(**kw), 0)
    assert e.value.status == status


def test_kv_shift_nothing_to_move_is_ok_without_gpu():
    """count = 0 and src = dst move nothing and launch nothing."""
    pb.pf_kv_shift(_shift_desc(count=0), 0)
    pb.pf_kv_shift(_shift_desc(dst=10), 0)


def _key_desc(**kw):
    d = pb.pf_key_desc()
    d.dtype, d.hidden = pb.PF_BF16, 64
    d.hidden_state, d.projection, d.key_out = 0x10000, 0x10000, 0x10000
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def _retrieval_desc(**kw):
    d = pb.pf_retrieval_desc()
    d.n_entries, d.lo, d.hi, d.token = 100, 0, 100, 7
    for f in ("query_key", "keys", "entry_token", "entry_pos", "entry_bound", "best",
              "similarity"):
        setattr(d, f, 0x10000)
    for k, v in kw.items():
        setattr(d, k, v)
    return d


def test_retrieval_rejects_bad_arguments():
    ws = pb.pf_retrieval_workspace_size()
    assert ws >= 1024 + 16 * 1024
    cases = [
        (lambda: pb.pf_retrieval_key(_key_desc(projection=None), 0x20000, ws), pb.PF_ERR_NULL),
        (lambda: pb.pf_retrieval_key(_key_desc(), 0x20000, ws - 1), pb.PF_ERR_WORKSPACE),
        (lambda: pb.pf_retrieval_key(_key_desc(dtype=4), 0x20000, ws), pb.PF_ERR_DTYPE),
        (lambda: pb.pf_retrieval_key(_key_desc(hidden=0), 0x20000, ws), pb.PF_ERR_SHAPE),
        (lambda: pb.pf_retrieval_key(_key_desc(), 0x20008, ws), pb.PF_ERR_ALIGN),
        (lambda: pb.pf_retrieve(_retrieval_desc(best=None), 0x20000, ws), pb.PF_ERR_NULL),
        (lambda: pb.pf_retrieve(_retrieval_desc(), 0, ws), pb.PF_ERR_WORKSPACE),
        (lambda: pb.pf_retrieve(_retrieval_desc(hi=101), 0x20000, ws), pb.PF_ERR_SHAPE),
        (lambda: pb.pf_retrieve(_retrieval_desc(lo=60, hi=50), 0x20000, ws), pb.PF_ERR_SHAPE),
        (lambda: pb.pf_retrieve(_retrieval_desc(keys=0x10004), 0x20000, ws), pb.PF_ERR_ALIGN),
        (lambda: pb.pf_retrieve(_retrieval_desc(entry_token=0x10008), 0x20000, ws),
         pb.PF_ERR_ALIGN),
        (lambda: pb.pf_retrieve(_retrieval_desc(entry_bound=0x10004), 0x20000, ws),
         pb.PF_ERR_ALIGN),
    ]
    for call, status in cases:
        with pytest.raises(pb.PfError) as e:
            call()
        assert e.value.status == status, pb.pf_last_error()


def test_prefix_match_rejects_bad_arguments():
    def desc(**kw):
        d = pb.pf_prefix_desc()
        d.prev, d.n_prev, d.next, d.n_next, d.lcp = 0x10000, 10, 0x10000, 12, 0x20000
        for k, v in kw.items():
            setattr(d, k, v)
        return d
    for kw, status in ((dict(lcp=None), pb.PF_ERR_NULL), (dict(n_prev=-1), pb.PF_ERR_SHAPE),
                       (dict(n_next=(1 << 30) + 1), pb.PF_ERR_SHAPE),
                       (dict(prev=None), pb.PF_ERR_NULL), (dict(next=None), pb.PF_ERR_NULL)):
        with pytest.raises(pb.PfError) as e:
            pb.pf_prefix_match(desc(**kw), 0)
        assert e.value.status == status


@pytest.mark.parametrize("kw,status", [
    (dict(parent=0), pb.PF_ERR_NULL),
    (dict(cu_nodes=0), pb.PF_ERR_NULL),
    (dict(mask_out=0), pb.PF_ERR_NULL),
    (dict(batch=0), pb.PF_ERR_SHAPE),
    (dict(total_nodes=0), pb.PF_ERR_SHAPE),
    (dict(max_nodes=0), pb.PF_ERR_SHAPE),
    (dict(max_nodes=129), pb.PF_ERR_SHAPE),
    (dict(mask_out=0x10008), pb.PF_ERR_ALIGN),
])
def test_tree_prepare_device_rejects_bad_arguments(kw, status):
    """Host checks of the device tree call: they return before any launch
    (here, with no GPU, before the library would notice there is none)."""
    a = dict(parent=0x10000, cu_nodes=0x10000, batch=2, total_nodes=9, max_nodes=8,
             depth_out=0, mask_out=0x10000)
    a.update(kw)
    with pytest.raises(pb.PfError) as e:
        pb.pf_tree_prepare_device(**a)
    assert e.value.status == status


def test_launch_fields_reach_the_library():
    """The launch fields sit after the workspace in pf_attn_desc, followed by
    the optional host copies of the lengths, and the stage request at the end
    of pf_lm_desc, as the header declares them."""
    names = [f[0] for f in pb.pf_attn_desc._fields_]
    assert names[-6:] == ["kernel", "splits", "rows_per_cta", "stages", "host_cu_nodes",
                          "host_prefix_len"]
    assert [f[0] for f in pb.pf_lm_desc._fields_][-1] == "stages"
