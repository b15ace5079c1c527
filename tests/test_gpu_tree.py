"""pf_tree_prepare_device (the device-side ancestor bitmaps of a batch of
proposal trees) against the oracle's parent walk and the host call, on
random, chain, star and 128-node trees, and its device checks on malformed
trees and sizes (error bits, no fault)."""
import numpy as np
import pytest
import torch

from oracle import tree as OT
from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I

pytestmark = pytest.mark.gpu


def _bits_to_sets(mask):
    """[N, 2] uint64 -> per node, the sorted list of set bit indices."""
    out = []
    for row in mask:
        bits = []
        for w in range(2):
            v = int(row[w])
            bits.extend(64 * w + i for i in range(64) if (v >> i) & 1)
        out.append(bits)
    return out


def _run(parents, max_nodes=None, cu=None):
    flat = np.concatenate([np.asarray(p, dtype=np.int32) for p in parents])
    if cu is None:
        cu = np.concatenate([[0], np.cumsum([len(p) for p in parents])]).astype(np.int32)
    T = int(flat.shape[0])
    max_nodes = max_nodes or max(len(p) for p in parents)
    d_parent = torch.from_numpy(flat).cuda()
    d_cu = torch.from_numpy(np.asarray(cu, dtype=np.int32)).cuda()
    # sentinel-filled outputs: rows the kernel skips keep the sentinel
    mask = torch.full((T, 2), -1, dtype=torch.int64, device="cuda")
    depth = torch.full((T,), -7, dtype=torch.int32, device="cuda")
    err = torch.zeros(1, dtype=torch.int32, device="cuda")
    pb.pf_tree_prepare_device(d_parent.data_ptr(), d_cu.data_ptr(), len(cu) - 1, T, max_nodes,
                              depth.data_ptr(), mask.data_ptr(), err.data_ptr(),
                              torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return (mask.cpu().numpy().view(np.uint64), depth.cpu().numpy(), int(err.item()))


def _trees():
    rng = np.random.default_rng(17)
    return [I.chain_tree(1), I.chain_tree(17), I.chain_tree(128),
            np.array([-1] + [0] * 63, dtype=np.int32),           # star
            I.random_tree(32, 3, rng), I.random_tree(128, 2, rng),
            I.chains_tree(64, 12, rng), I.chains_tree(128, 24, rng),
            I.random_tree(65, 5, rng)]


def test_matches_oracle_and_host_call():
    parents = _trees()
    mask, depth, err = _run(parents)
    assert err == 0
    off = 0
    for p in parents:
        n = len(p)
        got = _bits_to_sets(mask[off:off + n])
        assert got == OT.ancestor_mask_bits(p)
        assert np.array_equal(depth[off:off + n], OT.depths(p))
        hd, hm = pb.pf_tree_prepare(p)
        assert np.array_equal(mask[off:off + n], hm)
        assert np.array_equal(depth[off:off + n], hd)
        off += n


@pytest.mark.parametrize("bad", ["root-not-minus-one", "parent-not-before", "negative-parent",
                                 "self-parent"])
def test_malformed_tree_flags_and_keeps_self_bits(bad):
    good = I.chain_tree(10)
    p = good.copy()
    if bad == "root-not-minus-one":
        p[0] = 0
    elif bad == "parent-not-before":
        p[5] = 7
    elif bad == "negative-parent":
        p[3] = -2
    else:
        p[4] = 4
    assert not OT.validate(p)
    mask, depth, err = _run([good, p, good])
    assert err & pb.PF_DEVERR_TREE
    assert not err & pb.PF_DEVERR_BOUNDS
    # the malformed sequence: self bit only, depth -1; the others intact
    sets = _bits_to_sets(mask[10:20])
    assert sets == [[j] for j in range(10)]
    assert list(depth[10:20]) == [-1] * 10
    for off in (0, 20):
        assert _bits_to_sets(mask[off:off + 10]) == OT.ancestor_mask_bits(good)
        assert np.array_equal(depth[off:off + 10], OT.depths(good))


def test_sizes_outside_bounds_are_flagged_and_skipped():
    """A sequence with more nodes than max_nodes, and one whose cu_nodes
    reach past total_nodes: PF_DEVERR_BOUNDS, their rows untouched."""
    a, b, c = I.chain_tree(8), I.chain_tree(12), I.chain_tree(5)
    mask, depth, err = _run([a, b, c], max_nodes=10)
    assert err & pb.PF_DEVERR_BOUNDS
    assert (mask[8:20] == np.uint64(0xFFFFFFFFFFFFFFFF)).all()
    assert _bits_to_sets(mask[:8]) == OT.ancestor_mask_bits(a)
    assert _bits_to_sets(mask[20:25]) == OT.ancestor_mask_bits(c)
    cu = np.array([0, 8, 30], dtype=np.int32)   # the second sequence ends past T = 20
    mask, depth, err = _run([a, b], cu=cu)
    assert err & pb.PF_DEVERR_BOUNDS
    assert _bits_to_sets(mask[:8]) == OT.ancestor_mask_bits(a)
    assert (depth[8:] == -7).all()
