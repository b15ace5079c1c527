"""CUDA path (through the C ABI) against the fp64 oracle on seeded inputs.

Reduced sizes span several KV tiles, a ragged prefix tail, ragged vocabulary
and hidden tails, and both proposal tiles of large trees; the full-size
cases run the workloads' real shapes and check sampled outputs."""
import numpy as np
import pytest
import torch

from paper_2609_32166_gb300 import inputs as I
from tests.parity import Case

pytestmark = pytest.mark.gpu

W = I.WORKLOADS
SMALL = {
    "tiny-f32-chain8": W["tiny-f32-chain8"],
    "2b-chain16-small": I.scaled(W["2b-bf16-chain16"], layers=2, prefix=(300, 300), vocab=5000),
    "7b-tree64-small": I.scaled(W["7b-bf16-tree64"], layers=1, prefix=(1000, 1000), vocab=3000),
    "7b-batch8-paged-small": I.scaled(W["7b-bf16-batch8-paged"], layers=1, prefix=(100, 700),
                                      vocab=2000, hidden=512),
    "7b-32k-tree128-small": I.scaled(W["7b-bf16-32k-tree128"], layers=1, prefix=(2100, 2100),
                                     vocab=1000, hidden=256),
}


@pytest.mark.parametrize("name", sorted(SMALL))
def test_step_small(name):
    c = Case(SMALL[name], seed=0)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("seed", [1, 2])
def test_step_seeds(seed):
    c = Case(SMALL["7b-tree64-small"], seed=seed)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    c.check_attention(0, 0)
    c.check_lmhead(res)
    c.check_commit(res)


EDGE = {
    # root only: no drafts, a = 0, the tree tile holds one row
    "root-only": I.scaled(W["2b-bf16-chain16"], layers=1, prefix=(77, 77), nodes=1,
                          max_depth=0, vocab=700),
    # empty prefix: attention over the proposal's own ancestors only
    "empty-prefix": I.scaled(W["7b-bf16-tree64"], layers=1, prefix=(0, 0), vocab=900, hidden=256),
    # two proposal tiles (65 nodes), prefix one row past a tile boundary
    "65-nodes": I.scaled(W["7b-bf16-tree64"], layers=1, prefix=(129, 129), nodes=65,
                         max_depth=30, vocab=1300, hidden=264),
    # multi-head (G = 1), D = 64 bf16
    "mha-d64": I.scaled(W["7b-bf16-tree64"], layers=1, hq=4, hkv=4, d=64, prefix=(200, 200),
                        nodes=20, max_depth=8, vocab=515, hidden=128),
    # largest per-row group (G = 16), tiny vocabulary below one tile
    "g16-tiny-vocab": I.scaled(W["7b-bf16-tree64"], layers=1, hq=32, hkv=2, prefix=(64, 64),
                               nodes=9, max_depth=4, vocab=100, hidden=64),
    # 256 LM-head rows (2 x 128 nodes), paged
    "256-rows-paged": I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=2, prefix=(33, 300),
                               nodes=128, vocab=1000, hidden=192),
    # 192 rows of one KV head (two 128-row blocks in one CTA), one KV tile
    # (no split): the direct epilogue of the two-block kernel
    "two-blocks-one-tile": I.scaled(W["7b-bf16-tree64"], layers=1, hq=32, hkv=2, prefix=(0, 0),
                                    nodes=12, max_depth=5, vocab=300, hidden=64),
    # fp32 paged tree
    "f32-paged-tree": I.scaled(W["7b-bf16-batch8-paged"], dtype="f32", layers=2, batch=3,
                               hq=8, hkv=2, d=32, prefix=(5, 90), nodes=12, vocab=300,
                               hidden=96),
}


@pytest.mark.parametrize("name", sorted(EDGE))
def test_edge_cases(name):
    c = Case(EDGE[name], seed=5)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-batch8-paged-small"])
def test_mma_sync_kernel(name, monkeypatch):
    """The mma.sync attention kernel (selected with PF_ATTN_IMPL=mma) stays
    correct at D = 128, where the tcgen05 kernel is the default."""
    monkeypatch.setenv("PF_ATTN_IMPL", "mma")
    c = Case(SMALL[name], seed=6)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small"])
def test_64_token_tile_kernel(name, monkeypatch):
    """The tcgen05 kernel with 64-token tiles (PF_ATTN_IMPL=tc64), which the
    balanced batch mode and 256-row CTAs use, on 128-row CTAs too."""
    monkeypatch.setenv("PF_ATTN_IMPL", "tc64")
    c = Case(SMALL[name], seed=7)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        c.check_attention(l, 0)


@pytest.mark.parametrize("stages", ["2", "3"])
@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small"])
def test_128_token_tile_kernel(name, stages, monkeypatch):
    """The tcgen05 kernel with 128-token tiles and P in tensor memory
    (PF_ATTN_IMPL=tc128) also where a CTA holds few tiles, with both ring
    depths (3 stages: the merge inbox in the idle ring)."""
    monkeypatch.setenv("PF_ATTN_IMPL", "tc128")
    monkeypatch.setenv("PF_ATTN_W2_STAGES", stages)
    c = Case(SMALL[name], seed=9)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        c.check_attention(l, 0)


EDGE_128 = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                 "two-blocks-one-tile")}


@pytest.mark.parametrize("name", sorted(EDGE_128))
def test_128_token_tile_kernel_edges(name, monkeypatch):
    monkeypatch.setenv("PF_ATTN_IMPL", "tc128")
    c = Case(EDGE_128[name], seed=5)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)


@pytest.mark.parametrize("stages", ["2", "3"])
def test_128_token_tile_kernel_paged(stages, monkeypatch):
    """Paged cache (eight 16-token pages per 128-token tile, random page
    order, ragged last pages), two sequences with 128-node trees, on the
    128-token kernel (no workspace, so no balanced batch mode)."""
    monkeypatch.setenv("PF_ATTN_IMPL", "tc128")
    monkeypatch.setenv("PF_ATTN_W2_STAGES", stages)
    c = Case(EDGE["256-rows-paged"], seed=10, balanced=False)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-32k-tree128-small"])
def test_two_block_kernel_on_many_rows(name, monkeypatch):
    """Two 128-row blocks per CTA (PF_ATTN_BM=256) where a KV head has more
    than 256 rows, so several two-block CTAs share a head."""
    monkeypatch.setenv("PF_ATTN_BM", "256")
    c = Case(SMALL[name], seed=8)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("balanced", [False, True])
def test_batch_work_split(balanced):
    """Eight sequences with prefixes from 100 to 700 rows, with an attention
    workspace (tiles dealt out to the SMs in proportion to each sequence's
    length, partials merged by a second kernel) and without one (every
    sequence and KV head gets the same cluster)."""
    c = Case(SMALL["7b-batch8-paged-small"], seed=11, balanced=balanced)
    assert (c.vs.attn_ws is not None) == balanced
    assert c.vs.launches_per_step() == c.L * (2 if balanced else 1) + 2
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


def test_attention_workspace_contract():
    """The workspace query and the checks on a given workspace."""
    from paper_2609_32166_gb300 import binding as pb
    c = Case(SMALL["7b-batch8-paged-small"], seed=12)
    d = c.vs.attn_descs[0]
    need = pb.pf_verify_attention_workspace_size(d)
    assert need > 0 and need == c.vs.attn_ws_bytes
    d.workspace_bytes = need - 1
    with pytest.raises(pb.PfError) as e:
        pb.pf_verify_attention(d, 0)
    assert e.value.status == pb.PF_ERR_WORKSPACE
    d.workspace_bytes = need
    d.workspace = c.vs.attn_ws.data_ptr() + 8
    with pytest.raises(pb.PfError) as e:
        pb.pf_verify_attention(d, 0)
    assert e.value.status == pb.PF_ERR_ALIGN
    d.workspace = c.vs.attn_ws.data_ptr()
    # a single sequence needs none (its KV heads and row blocks share clusters)
    one = Case(SMALL["7b-tree64-small"], seed=12)
    assert pb.pf_verify_attention_workspace_size(one.vs.attn_descs[0]) == 0
    assert one.vs.attn_ws is None


def test_batch_beyond_balanced_groups():
    """More (sequence, KV head) groups than SMs: no workspace is asked for
    and every sequence goes through the cluster path."""
    import torch as _t
    sms = _t.cuda.get_device_properties(0).multi_processor_count
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=sms // 4 + 2, prefix=(20, 150),
                 nodes=6, vocab=300, hidden=64)
    c = Case(w, seed=13)
    assert c.vs.attn_ws is None
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in sorted({0, 1, w.batch // 2, w.batch - 1}):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("impl", ["default", "tc128"])
def test_mixed_tree_sizes(impl, monkeypatch):
    """Sequences of 1, 17 and 128 nodes in one batch (variable cu_nodes), on
    the default path (balanced batch mode) and on the 128-token kernel."""
    if impl == "tc128":
        monkeypatch.setenv("PF_ATTN_IMPL", "tc128")
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=3, prefix=(50, 400), nodes=128,
                 vocab=640, hidden=128)
    rng = np.random.default_rng(9)
    parents = [I.chain_tree(1), I.random_tree(17, 3, rng), I.chains_tree(128, 24, rng)]
    prefix = np.array([400, 50, 129], dtype=np.int32)
    ends = np.array([0, 16, 127], dtype=np.int32)
    max_seq = int(prefix.max()) + 128
    per_seq = -(-max_seq // I.PAGE_SIZE)
    pt = rng.permutation(per_seq * 3).astype(np.int32).reshape(3, per_seq)
    b = I.Batch(w, 7, parents, prefix, ends, pt, per_seq * 3, max_seq)
    c = Case(w, batch=b, balanced=impl == "default")
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(3):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


def test_deterministic_and_repeatable():
    c = Case(SMALL["7b-batch8-paged-small"], seed=3)
    c.vs.step()
    a = c.vs.attn_out.clone()
    r1 = c.vs.results()
    c.vs.step()
    r2 = c.vs.results()
    assert torch.equal(a, c.vs.attn_out)
    for k in ("argmax", "accept_len", "path", "out_tokens", "new_len"):
        assert np.array_equal(r1[k], r2[k])
    # the LM-head workspace is left zeroed by every call
    assert int(c.vs.workspace.count_nonzero().item()) == 0


def test_commit_capacity_flag_without_fault():
    """A page-table hole where a committed row should go: the kernel skips the
    row and reports PF_DEVERR_CAPACITY instead of writing outside the cache."""
    from paper_2609_32166_gb300 import binding as pb
    c = Case(SMALL["7b-batch8-paged-small"], seed=4)
    c.vs.attention(0)
    c.vs.lmhead()
    torch.cuda.synchronize()
    P = int(c.batch.prefix_lens[0])
    c.vs.page_table[0, P // I.PAGE_SIZE] = -1
    c.vs.commit()
    res = c.vs.results()
    assert res["err"] & pb.PF_DEVERR_CAPACITY


# ---------------------------------------------------------------------------
# full workload sizes (sampled checks)
# ---------------------------------------------------------------------------
FULL = {
    "2b-bf16-chain16": 28,
    "7b-bf16-tree64": 2,
    "7b-bf16-batch8-paged": 1,
    "7b-bf16-32k-tree128": 1,
}


@pytest.mark.parametrize("name", sorted(FULL))
def test_full_size_sampled(name):
    w = W[name]
    c = Case(w, seed=0, layers=FULL[name])
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    layers = sorted({0, c.L // 2, c.L - 1})
    for l in layers:
        for s in sorted({0, w.batch - 1}):
            n = int(c.batch.cu_nodes[s + 1] - c.batch.cu_nodes[s])
            nodes = sorted({0, n - 1, n // 2, int(c.batch.forced_end[s])})
            c.check_attention(l, s, nodes=nodes)
    flagged = c.check_lmhead(res)
    print(f"{name}: flagged near-tie nodes {flagged}/{c.batch.total_nodes}")
    c.check_commit(res, layers=layers)
