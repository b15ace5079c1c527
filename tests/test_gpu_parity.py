"""CUDA path (through the C ABI) against the fp64 oracle on seeded inputs.

Reduced sizes span several KV tiles, a ragged prefix tail, ragged vocabulary
and hidden tails, and both proposal tiles of large trees; the full-size
cases run the workloads' real shapes and check sampled outputs."""
import numpy as np
import pytest
import torch

from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I
from tests.parity import Case

MMA = dict(kernel=pb.PF_ATTN_KERNEL_MMA)
TC64 = dict(kernel=pb.PF_ATTN_KERNEL_TC64)
TC128 = dict(kernel=pb.PF_ATTN_KERNEL_TC128)
PAIR = dict(kernel=pb.PF_ATTN_KERNEL_PAIR)

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


# ---------------------------------------------------------------------------
# the SM-pair kernel (2-SM MMA, each CTA holding half of every K/V tile)
# ---------------------------------------------------------------------------
EDGE_PAIR = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                  "256-rows-paged", "two-blocks-one-tile")}


@pytest.mark.parametrize("balanced", [False, True])
@pytest.mark.parametrize("name", sorted(EDGE_PAIR))
def test_pair_kernel_edges(name, balanced):
    """Root only (the odd CTA of the pair has no rows), no prefix (one tile),
    65 nodes with a one-row last prefix tile, G = 16 (the odd CTA holds one
    node), 128-node paged trees, one tile for 192 rows; cluster mode and the
    balanced batch mode (the latter only changes batches)."""
    c = Case(EDGE_PAIR[name], seed=5, balanced=balanced, attn_launch=PAIR)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("splits", [1, 2, 3, 8])
@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-32k-tree128-small",
                                  "7b-batch8-paged-small"])
def test_pair_kernel_splits(name, splits):
    """Pairs per cluster from 1 to 8 (cluster widths 2 to 16) on the three 7B
    shapes, paged batch included (cluster mode: no workspace), every node."""
    c = Case(SMALL[name], seed=14, balanced=False, attn_launch=dict(PAIR, splits=splits))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("launch", ["tc64", "pair"])
def test_splits_without_tiles(launch):
    """A split count above a sequence's tile count: with 8 splits, a
    sequence whose prefix is 20 rows has 2 tiles, so 6 splits (tc64) or 6
    pairs (pair kernel) of its cluster get no tile and contribute zero
    partials with lse = -inf to the merge."""
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=3, prefix=(20, 1500), nodes=20,
                 max_depth=6, vocab=600, hidden=128)
    rng = np.random.default_rng(21)
    parents = [I.random_tree(20, 3, rng) for _ in range(3)]
    prefix = np.array([20, 1500, 700], dtype=np.int32)
    ends = np.array([5, 11, 19], dtype=np.int32)
    max_seq = int(prefix.max()) + 20
    per_seq = -(-max_seq // I.PAGE_SIZE)
    pt = rng.permutation(per_seq * 3).astype(np.int32).reshape(3, per_seq)
    b = I.Batch(w, 3, parents, prefix, ends, pt, per_seq * 3, max_seq)
    tile = 64 if launch == "tc64" else 128
    n_tiles = -(-int(prefix[0]) // tile) + 1
    assert n_tiles < 8   # the case under test occurs
    launch_fields = dict(TC64, rows_per_cta=128) if launch == "tc64" else dict(PAIR)
    c = Case(w, batch=b, balanced=False, attn_launch=dict(launch_fields, splits=8))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(3):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


def test_two_block_kernel_one_tile():
    """192 rows of one KV head in one two-block CTA of the 64-token kernel,
    one KV tile (no split): that kernel's direct epilogue."""
    c = Case(EDGE["two-blocks-one-tile"], seed=5, attn_launch=dict(TC64, rows_per_cta=256))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    c.check_attention(0, 0)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-batch8-paged-small"])
def test_mma_sync_kernel(name):
    """The mma.sync attention kernel (kernel = PF_ATTN_KERNEL_MMA) stays
    correct at D = 128, where the tcgen05 kernels are the default."""
    c = Case(SMALL[name], seed=6, attn_launch=MMA)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small"])
def test_64_token_tile_kernel(name):
    """The tcgen05 kernel with 64-token tiles (PF_ATTN_KERNEL_TC64), its
    balanced batch mode and 256-row CTAs, on 128-row CTAs too."""
    c = Case(SMALL[name], seed=7, attn_launch=dict(TC64, rows_per_cta=128))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        c.check_attention(l, 0)


@pytest.mark.parametrize("stages", [2, 3])
@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small"])
def test_128_token_tile_kernel(name, stages):
    """The tcgen05 kernel with 128-token tiles and P in tensor memory
    (PF_ATTN_KERNEL_TC128) also where a CTA holds few tiles, with both ring
    depths (3 stages: the merge inbox in the idle ring)."""
    c = Case(SMALL[name], seed=9, attn_launch=dict(TC128, stages=stages))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        c.check_attention(l, 0)


EDGE_128 = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                 "two-blocks-one-tile")}


@pytest.mark.parametrize("name", sorted(EDGE_128))
def test_128_token_tile_kernel_edges(name):
    c = Case(EDGE_128[name], seed=5, attn_launch=TC128)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)


@pytest.mark.parametrize("stages", [2, 3])
def test_128_token_tile_kernel_paged(stages):
    """Paged cache (eight 16-token pages per 128-token tile, random page
    order, ragged last pages), two sequences with 128-node trees, on the
    128-token kernel (no workspace, so no balanced batch mode)."""
    c = Case(EDGE["256-rows-paged"], seed=10, balanced=False,
             attn_launch=dict(TC128, stages=stages))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-32k-tree128-small"])
def test_two_block_kernel_on_many_rows(name):
    """Two 128-row blocks per CTA (64-token kernel, rows_per_cta = 256) where
    a KV head has more than 256 rows, so several two-block CTAs share a head."""
    c = Case(SMALL[name], seed=8, attn_launch=dict(TC64, rows_per_cta=256))
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("kernel", ["auto", "pair"])
@pytest.mark.parametrize("balanced", [False, True])
def test_batch_work_split(balanced, kernel):
    """Eight sequences with prefixes from 100 to 700 rows, with an attention
    workspace (tiles dealt out to the SMs -- or SM pairs -- in proportion to
    each sequence's length, partials merged by a second kernel) and without
    one (every sequence and KV head gets the same cluster); on the automatic
    choice and on the SM-pair kernel."""
    c = Case(SMALL["7b-batch8-paged-small"], seed=11, balanced=balanced,
             attn_launch=PAIR if kernel == "pair" else None)
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


@pytest.mark.parametrize("impl", ["default", "tc128", "pair-clusters"])
def test_mixed_tree_sizes(impl):
    """Sequences of 1, 17 and 128 nodes in one batch (variable cu_nodes), on
    the default path (balanced batch mode on SM pairs), on the 128-token
    kernel and on SM pairs in cluster mode."""
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
    launch = {"default": None, "tc128": TC128, "pair-clusters": PAIR}[impl]
    c = Case(w, batch=b, balanced=impl == "default", attn_launch=launch)
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
# full workload sizes, in the launch configuration bench.py times
# ---------------------------------------------------------------------------
FULL = {
    "2b-bf16-chain16": 28,
    "7b-bf16-tree64": 2,
    "7b-bf16-batch8-paged": 1,
    "7b-bf16-32k-tree128": 1,
}
FULL_CASES = [("2b-bf16-chain16", 0), ("7b-bf16-tree64", 0), ("7b-bf16-tree64", 1),
              ("7b-bf16-batch8-paged", 0), ("7b-bf16-32k-tree128", 0),
              ("7b-bf16-32k-tree128", 1)]


@pytest.fixture(scope="module")
def oracle_pool():
    from tests.oracle_pool import make_pool
    pool = make_pool()
    yield pool
    pool.shutdown()


@pytest.mark.parametrize("name,seed", FULL_CASES)
def test_full_size(name, seed, oracle_pool):
    """The workloads' real shapes with the library's automatic launch choice
    (the balanced batch mode for the batch): every node and head of layer 0
    of every sequence against the oracle (for the 32K tree's second seed,
    four sampled nodes), sampled nodes of the middle and last layer, then the
    LM head, acceptance and commit."""
    import time
    from tests.oracle_pool import oracle_attention_nodes
    w = W[name]
    t0 = time.time()
    c = Case(w, seed=seed, layers=FULL[name])
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    every = not (name == "7b-bf16-32k-tree128" and seed == 1)
    errs = []
    for s in range(w.batch):
        n = int(c.batch.cu_nodes[s + 1] - c.batch.cu_nodes[s])
        nodes = range(n) if every else sorted({0, n - 1, n // 2, int(c.batch.forced_end[s])})
        ref = oracle_attention_nodes(oracle_pool, w, seed, 0, s, nodes)
        errs.append(c.compare_attention(0, s, ref))
    layers = sorted({0, c.L // 2, c.L - 1})
    for l in layers[1:]:
        for s in sorted({0, w.batch - 1}):
            n = int(c.batch.cu_nodes[s + 1] - c.batch.cu_nodes[s])
            c.check_attention(l, s, nodes=sorted({0, n - 1, n // 2, int(c.batch.forced_end[s])}))
    flagged = c.check_lmhead(res)
    c.check_commit(res, layers=layers)
    print(f"{name} seed {seed}: layer-0 max error {max(errs):.2e} over "
          f"{'every node' if every else 'sampled nodes'}, flagged near-tie nodes "
          f"{flagged}/{c.batch.total_nodes}, {time.time() - t0:.0f} s")
