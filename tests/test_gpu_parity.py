"""CUDA path (through the C ABI) against the fp64 oracle on seeded inputs.

Reduced sizes span several KV tiles, a ragged prefix tail, ragged vocabulary
and hidden tails, and both proposal tiles of large trees; the full-size
cases run the workloads' real shapes and check sampled outputs."""
import numpy as np
import pytest
import torch

from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I
from oracle import attention as OA
from tests.parity import Case, values

MMA = dict(kernel=pb.PF_ATTN_KERNEL_MMA)
TC64 = dict(kernel=pb.PF_ATTN_KERNEL_TC64)
TC128 = dict(kernel=pb.PF_ATTN_KERNEL_TC128)
PAIR = dict(kernel=pb.PF_ATTN_KERNEL_PAIR)
STREAM = dict(kernel=pb.PF_ATTN_KERNEL_STREAM)
BATCH = dict(kernel=pb.PF_ATTN_KERNEL_BATCH)

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
# the SM-pair kernel (2-SM MMA, each CTA holding half of every K/V tile; all
# groups' tiles cut into one equal range per SM pair)
# ---------------------------------------------------------------------------
EDGE_PAIR = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                  "256-rows-paged", "two-blocks-one-tile")}


@pytest.mark.parametrize("name", sorted(EDGE_PAIR))
def test_pair_kernel_edges(name):
    """Root only (the odd CTA of the pair has no rows, most pairs no tile),
    no prefix (one tile), 65 nodes with a one-row last prefix tile, G = 16
    (the odd CTA holds one node), 128-node paged trees, one tile for 192
    rows."""
    c = Case(EDGE_PAIR[name], seed=5, attn_launch=PAIR)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-32k-tree128-small",
                                  "7b-batch8-paged-small"])
def test_pair_kernel_shapes(name):
    """The three 7B shapes, every node: groups cut into pieces over many
    pairs (the 32K tree's groups span ~10 ranges each), pieces merged."""
    c = Case(SMALL[name], seed=14, attn_launch=PAIR)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)


def test_pair_kernel_many_groups():
    """More groups than SM pairs: 40 sequences x 4 KV heads, 160 groups of
    1..7 tiles, so one pair's range holds several whole groups besides the
    pieces at its ends (whole groups write their output directly); 6 nodes
    per sequence keep the batch within the LM head's 256 rows."""
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=40, prefix=(20, 700), nodes=6,
                 max_depth=5, vocab=300, hidden=64)
    c = Case(w, seed=15, attn_launch=PAIR)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("kernel", ["pair", "stream", "batch"])
def test_continuous_split_needs_the_workspace(kernel):
    c = Case(SMALL["7b-tree64-small"], seed=16, balanced=False)
    d = c.vs.attn_descs[0]
    d.kernel = {"pair": pb.PF_ATTN_KERNEL_PAIR, "stream": pb.PF_ATTN_KERNEL_STREAM,
                "batch": pb.PF_ATTN_KERNEL_BATCH}[kernel]
    assert pb.pf_verify_attention_launches(d) == 0
    with pytest.raises(pb.PfError) as e:
        pb.pf_verify_attention(d, 0)
    assert e.value.status == pb.PF_ERR_WORKSPACE


# ---------------------------------------------------------------------------
# the continuous-split kernel (128-token tiles, one CTA per SM, all groups'
# tiles cut into one equal range per SM)
# ---------------------------------------------------------------------------
EDGE_STREAM = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                    "256-rows-paged", "two-blocks-one-tile")}


@pytest.mark.parametrize("name", sorted(EDGE_STREAM))
def test_stream_kernel_edges(name):
    c = Case(EDGE_STREAM[name], seed=5, attn_launch=STREAM)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small",
                                  "7b-batch8-paged-small"])
def test_stream_kernel_shapes(name):
    """Single sequences and the paged batch, every node: groups cut into
    pieces over many SMs (the 32K tree's groups span ~6 ranges each)."""
    c = Case(SMALL[name], seed=17, attn_launch=STREAM)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)


def test_stream_kernel_many_groups():
    """120 groups (30 sequences x 4 KV heads): ranges of whole groups and
    pieces; the most the kernel takes is 128."""
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=30, prefix=(20, 900), nodes=8,
                 max_depth=5, vocab=300, hidden=64)
    c = Case(w, seed=18, attn_launch=STREAM)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


# ---------------------------------------------------------------------------
# the batch kernel (128-token tiles, one CTA per SM, each group spread over
# CTAs in proportion to its tiles, the last piece merging in the kernel)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("name", sorted(EDGE_STREAM))
def test_batch_kernel_edges(name):
    c = Case(EDGE_STREAM[name], seed=6, attn_launch=BATCH)
    assert c.vs.launches_per_step() == c.L + 2  # no merge kernel
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["2b-chain16-small", "7b-tree64-small", "7b-32k-tree128-small",
                                  "7b-batch8-paged-small"])
def test_batch_kernel_shapes(name):
    """Every node: single sequences (a group's tiles spread over up to all
    SMs, many pieces per merge) and the paged batch."""
    c = Case(SMALL[name], seed=19, attn_launch=BATCH)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)


def test_batch_kernel_many_groups():
    """144 groups (36 sequences x 4 KV heads, 252 proposal rows) of 1..9
    tiles on the SMs: most groups whole on one CTA, the longest in pieces."""
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=36, prefix=(20, 900), nodes=7,
                 max_depth=5, vocab=300, hidden=64)
    c = Case(w, seed=20, attn_launch=BATCH)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(w.batch):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


def test_batch_kernel_tickets_need_no_initialisation():
    """A workspace full of 0xff bytes (and one left by other calls), then a
    CUDA graph of the layer replayed three times with the same epoch: every
    result equals the eager call's (the last piece resets its ticket)."""
    c = Case(SMALL["7b-batch8-paged-small"], seed=21, attn_launch=BATCH)
    c.vs.attn_ws.fill_(0xff)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(c.w.batch):
        c.check_attention(0, s)
    ref = c.vs.attn_out.clone()
    stream = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        c.vs.attention(0, torch.cuda.current_stream().cuda_stream)
    for _ in range(3):
        c.vs.attn_out.zero_()
        with torch.cuda.stream(stream):
            g.replay()
        stream.synchronize()
        assert torch.equal(c.vs.attn_out[0], ref[0])
    assert c.vs.results()["err"] == 0


def test_splits_without_tiles():
    """A split count above a sequence's tile count: with 8 splits, a
    sequence whose prefix is 20 rows has 2 64-token tiles, so 6 splits of
    its cluster get no tile and contribute zero partials with lse = -inf to
    the merge."""
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
    n_tiles = -(-int(prefix[0]) // 64) + 1
    assert n_tiles < 8   # the case under test occurs
    c = Case(w, batch=b, balanced=False, attn_launch=dict(TC64, rows_per_cta=128, splits=8))
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


# ---------------------------------------------------------------------------
# two 128-row blocks per CTA on 128-token tiles (PF_ATTN_KERNEL_TWO_BLOCK):
# K and V in separate ring units, each block's P written over its S columns
# ---------------------------------------------------------------------------
TWO_BLOCK = dict(kernel=pb.PF_ATTN_KERNEL_TWO_BLOCK)
EDGE_2BLK = {k: EDGE[k] for k in ("root-only", "empty-prefix", "65-nodes", "g16-tiny-vocab",
                                  "256-rows-paged", "two-blocks-one-tile")}


@pytest.mark.parametrize("name", sorted(EDGE_2BLK))
def test_two_block_128_kernel_edges(name):
    """Root only (one row, block B empty), no prefix, two proposal tiles with
    a prefix one row past a tile boundary, G = 16, 256 rows on a paged cache,
    and 192 rows in one tile (the direct epilogue)."""
    c = Case(EDGE_2BLK[name], seed=5, balanced=False, attn_launch=TWO_BLOCK)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("name", ["7b-tree64-small", "7b-32k-tree128-small",
                                  "7b-batch8-paged-small"])
def test_two_block_128_kernel(name):
    """448 and 896 rows per KV head (two and four two-block CTAs per head),
    and eight sequences of 224 rows on a paged cache whose shortest prefixes
    leave some splits of a cluster without tiles."""
    c = Case(SMALL[name], seed=12, balanced=False, attn_launch=TWO_BLOCK)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for l in range(c.L):
        for s in range(c.w.batch):
            c.check_attention(l, s)


@pytest.mark.parametrize("host_lengths", ["given", "absent", "stale"])
def test_two_block_128_kernel_teams(host_lengths):
    """Eight sequences with prefixes from 100 to 1500 rows: with the host's
    copies of the lengths (teams of a cluster's CTAs per group, sized by the
    groups' tiles), without them (one group per cluster), and with copies
    that disagree with the device arrays (a plan made for other lengths
    still covers every tile once)."""
    w = I.scaled(SMALL["7b-batch8-paged-small"], prefix=(100, 1500))
    c = Case(w, seed=15, balanced=False, attn_launch=TWO_BLOCK)
    if host_lengths == "absent":
        for d in c.vs.attn_descs:
            d.host_cu_nodes = d.host_prefix_len = None
    elif host_lengths == "stale":
        c.vs.h_prefix_len[:] = c.vs.h_prefix_len[::-1].copy()
    c.vs.attention(0)
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(w.batch):
        c.check_attention(0, s)


@pytest.mark.parametrize("splits", [1, 2, 3, 4, 5, 6, 7, 8, 9, 16])
def test_two_block_128_kernel_splits(splits):
    """Every cluster width from one CTA (no merge) to 16 (wider than the
    nine tiles: splits without tiles merge a zero partial)."""
    c = Case(SMALL["7b-tree64-small"], seed=13, balanced=False,
             attn_launch=dict(TWO_BLOCK, splits=splits))
    c.vs.attention(0)
    res = c.vs.results()
    assert res["err"] == 0
    c.check_attention(0, 0)


@pytest.mark.parametrize("kernel", ["tc128", "two_block"])
@pytest.mark.parametrize("layout", ["contiguous", "paged"])
def test_growing_scores_rescale_the_accumulator(kernel, layout):
    """Prefix keys scaled up along the sequence (x1 to x12), so that within a
    split's six tiles the row maximum outgrows the running one by more than
    the kernels' lazy rescale threshold (2^8) and the accumulated O and row
    sum are rescaled; checked against the oracle on the same scaled keys."""
    w = I.scaled(SMALL["7b-tree64-small"], layout=layout, prefix=(1500, 1500))
    launch = dict({"tc128": TC128, "two_block": TWO_BLOCK}[kernel], splits=2)
    c = Case(w, seed=14, balanced=False, attn_launch=launch)
    b = c.batch
    pk, pv = I.layer_prefix_kv(w, b, 0, 0)
    P = pk.shape[1]
    ramp = np.linspace(1.0, 12.0, P, dtype=np.float32)[None, :, None]
    pk2 = I.round_to_bf16_bits(values(pk, "bf16") * ramp)
    ck = np.zeros(I.cache_shape(w, b), dtype=np.uint16)
    I.place_prefix(w, b, ck, 0, pk2)
    c.vs.cache_k[0] = torch.from_numpy(ck.view(np.int16)).view(torch.bfloat16).to(
        c.vs.cache_k.device)
    c.vs.attention(0)
    res = c.vs.results()
    assert res["err"] == 0
    c0, c1 = int(b.cu_nodes[0]), int(b.cu_nodes[1])
    q = values(I.layer_q(w, b, 0), "bf16")[c0:c1]
    tk, tv = (values(x, "bf16")[c0:c1] for x in I.layer_tree_kv(w, b, 0))
    ref = OA.tree_attention(q, values(pk2, "bf16"), values(pv, "bf16"), tk, tv, b.parents[0])
    got = c.vs.attn_out[0, c0:c1].float().cpu().numpy().astype(np.float64)
    assert np.isfinite(got).all()
    err = float(np.abs(got - ref).max())
    assert err <= 2e-2, err


@pytest.mark.parametrize("kernel", ["auto", "two_block"])
@pytest.mark.parametrize("nodes", [2, 17, 63, 64, 127])
def test_node_count_sweep(nodes, kernel):
    """Proposal sizes around the 64- and 128-token tile edges (1, 9, 65 and
    128 nodes are among the edge cases), two sequences with prefixes of 448
    and 515 rows (a multiple of 64 but not of 128; a multiple of neither),
    every node and head, then the LM head, acceptance and commit."""
    w = I.scaled(W["7b-bf16-tree64"], layers=1, batch=2, prefix=(333, 517), nodes=nodes,
                 max_depth=min(nodes - 1, 12), vocab=700, hidden=128)
    launch = None if kernel == "auto" else TWO_BLOCK
    c = Case(w, seed=16, balanced=False, attn_launch=launch)
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in range(w.batch):
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


@pytest.mark.parametrize("kernel,balanced", [("auto", True), ("auto", False), ("tc64", False),
                                             ("tc64", True), ("stream", True), ("pair", True),
                                             ("batch", True)])
def test_batch_work_split(balanced, kernel):
    """Eight sequences with prefixes from 100 to 700 rows: the automatic
    choice (clusters of 128-row CTAs, no workspace even when one is
    offered); the 64-token kernel's two-block CTAs without a workspace
    (every sequence and KV head gets the same cluster) and with one (tiles
    dealt out to the SMs in proportion to each sequence's length); the
    continuous split on SMs and on SM pairs (partials merged by a second
    kernel); the batch kernel (pieces in proportion to each sequence's
    tiles, merged by the last piece in the same launch)."""
    launch = {"auto": None, "tc64": TC64, "stream": STREAM, "pair": PAIR, "batch": BATCH}[kernel]
    c = Case(SMALL["7b-batch8-paged-small"], seed=11, balanced=balanced, attn_launch=launch)
    assert (c.vs.attn_ws is not None) == (balanced and kernel != "auto")
    merge_kernel = balanced and kernel in ("tc64", "stream", "pair")
    assert c.vs.launches_per_step() == c.L * (2 if merge_kernel else 1) + 2
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
    c = Case(SMALL["7b-batch8-paged-small"], seed=12, attn_launch=TC64)
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
    # the automatic choice needs none (its KV heads and row blocks share
    # clusters), the continuous-split and batch kernels one for any batch
    one = Case(SMALL["7b-tree64-small"], seed=12)
    assert pb.pf_verify_attention_workspace_size(one.vs.attn_descs[0]) == 0
    assert one.vs.attn_ws is None
    auto = Case(SMALL["7b-batch8-paged-small"], seed=12)
    assert pb.pf_verify_attention_workspace_size(auto.vs.attn_descs[0]) == 0
    for k in (pb.PF_ATTN_KERNEL_PAIR, pb.PF_ATTN_KERNEL_STREAM, pb.PF_ATTN_KERNEL_BATCH):
        one_k = Case(SMALL["7b-tree64-small"], seed=12, attn_launch=dict(kernel=k))
        assert pb.pf_verify_attention_workspace_size(one_k.vs.attn_descs[0]) > 0


def test_batch_beyond_balanced_groups():
    """More (sequence, KV head) groups than SMs on the 64-token kernel: its
    balanced batch mode does not apply, no workspace is asked for and every
    sequence goes through the cluster path."""
    import torch as _t
    sms = _t.cuda.get_device_properties(0).multi_processor_count
    w = I.scaled(W["7b-bf16-batch8-paged"], layers=1, batch=sms // 4 + 2, prefix=(20, 150),
                 nodes=6, vocab=300, hidden=64)
    c = Case(w, seed=13, attn_launch=TC64)
    assert c.vs.attn_ws is None
    c.vs.step()
    res = c.vs.results()
    assert res["err"] == 0
    for s in sorted({0, 1, w.batch // 2, w.batch - 1}):
        c.check_attention(0, s)
    c.check_lmhead(res)
    c.check_commit(res)


@pytest.mark.parametrize("impl", ["default", "batch", "tc64-balanced", "stream"])
def test_mixed_tree_sizes(impl):
    """Sequences of 1, 17 and 128 nodes in one batch (variable cu_nodes), on
    the default path (clusters), on the batch kernel, on the 64-token
    kernel's balanced batch mode and on the continuous split."""
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
    launch = {"default": None, "batch": BATCH, "tc64-balanced": TC64, "stream": STREAM}[impl]
    c = Case(w, batch=b, attn_launch=launch)
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
