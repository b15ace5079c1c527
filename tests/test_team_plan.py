"""The two-block kernel's team plan (host code): pf_verify_attention_team_plan
with a given table of how many clusters fit on the GPU, so no GPU is needed.

Checked on random batches: every (sequence, KV head, pair of row blocks)
group that holds nodes is one team of consecutive CTAs inside one cluster,
its pieces 0..k-1 each exactly once at cluster ranks base..base+k-1; no
other group appears; the launch is whole clusters, no more than fit and no
more CTAs than SMs, numbered longest piece first; the reported longest
piece is the plan's and beats the one-group clusters it was asked to
beat."""
import math

import numpy as np
import pytest

from paper_2609_32166_gb300 import binding as pb

GB300_LIKE = [0] + [min(152 // s, {8: 15, 10: 13, 12: 11, 14: 9, 16: 8}.get(s, 152))
                    for s in range(1, 17)]


def decode(e):
    e = int(e)
    return e & 0xFFF, (e >> 12) & 31, (e >> 17) & 31, (e >> 22) & 31


def tiles(P, nn):
    return (P + 127) // 128 + (nn + 127) // 128


def check_plan(cu, P, hkv, G, max_nodes, max_prefix, sms, table, uniform):
    st, entries, s, ctas, span = pb.pf_verify_attention_team_plan(
        cu, P, hkv, G, max_nodes, max_prefix, sms, table, uniform)
    assert st in (0, 1)
    if st == 0:
        return None
    nb = 2 * (128 // G)
    pairs = math.ceil(max_nodes / nb)
    assert s >= 2 and s % 2 == 0 and s <= 16
    assert ctas % s == 0 and 0 < ctas <= min(sms, pb.PF_TEAM_MAX_CTAS)
    assert ctas // s <= table[s]
    assert not entries[ctas:].any()
    teams = {}
    for i in range(ctas):
        g, part, k, base = decode(entries[i])
        if k == 0:
            continue
        c, rank = divmod(i, s)
        assert 0 <= part < k and rank == base + part and base + k <= s
        t = teams.setdefault(g, {"cluster": c, "k": k, "base": base, "parts": set()})
        assert (t["cluster"], t["k"], t["base"]) == (c, k, base)
        assert part not in t["parts"]
        t["parts"].add(part)
    want = {}
    for b in range(len(P)):
        nn = int(cu[b + 1] - cu[b])
        for g in range(hkv):
            for rb in range(math.ceil(nn / nb)):
                want[(b * hkv + g) * pairs + rb] = tiles(int(P[b]), nn)
    assert set(teams) == set(want)
    longest = 0
    for g, t in teams.items():
        assert t["parts"] == set(range(t["k"]))
        longest = max(longest, math.ceil(want[g] / t["k"]))
    assert span == longest
    assert span < math.ceil(max(want.values()) / uniform)
    # no cluster holds more CTAs than it has; every cluster of the launch
    # holds a team; clusters come longest piece first (they start in order)
    used, piece = {}, {}
    for g, t in teams.items():
        c = t["cluster"]
        used[c] = used.get(c, 0) + t["k"]
        piece[c] = max(piece.get(c, 0), math.ceil(want[g] / t["k"]))
    assert all(v <= s for v in used.values())
    assert sorted(used) == list(range(ctas // s))
    assert all(piece[c] >= piece[c + 1] for c in range(ctas // s - 1))
    return s, ctas, span


@pytest.mark.parametrize("seed", range(40))
def test_random_batches(seed):
    rng = np.random.default_rng(seed)
    B = int(rng.integers(2, 17))
    G = int(rng.choice([1, 6, 7, 16]))
    hkv = int(rng.choice([1, 2, 4, 8]))
    nodes = rng.integers(1, 129, size=B)
    P = rng.integers(0, 8001, size=B).astype(np.int32)
    cu = np.concatenate([[0], np.cumsum(nodes)]).astype(np.int32)
    table = GB300_LIKE if seed % 2 == 0 else [0] + [152 // s for s in range(1, 17)]
    check_plan(cu, P, hkv, G, int(nodes.max()), int(P.max()), 152, table, 2)


def test_headline_batch():
    """The 8-sequence batch's lengths (prefixes 2232..5767, 32-node trees,
    G = 7, 4 KV heads): one group per cluster leaves 12 tiles on the longest
    CTAs (4 CTAs per group); the plan gets to at most 11 in clusters that fit,
    against 8 for an even split over 152 SMs."""
    P = np.array([2232, 5480, 5767, 3188, 5723, 3995, 5681, 3922], np.int32)
    cu = np.arange(0, 33 * 8, 32, dtype=np.int32)[:9]
    got = check_plan(cu, P, 4, 7, 32, int(P.max()), 152, GB300_LIKE, 4)
    assert got is not None
    s, ctas, span = got
    total = sum(tiles(int(p), 32) for p in P) * 4
    assert math.ceil(total / 152) <= span <= 11


def test_declines_where_it_cannot_beat_the_uniform_clusters():
    # one sequence, one KV head, one pair of row blocks: a single group
    st = pb.pf_verify_attention_team_plan([0, 32], [4096], 1, 7, 32, 4096, 152, GB300_LIKE, 16)[0]
    assert st == 0
    # equal groups that the one-group clusters already split finely
    cu = np.array([0, 64], np.int32)
    st = pb.pf_verify_attention_team_plan(cu, [4096], 4, 7, 64, 4096, 152, GB300_LIKE, 16)[0]
    assert st == 0


def test_rejects_inconsistent_lengths_and_bad_arguments():
    cu = np.array([0, 10, 10], np.int32)  # a sequence without nodes
    assert pb.pf_verify_attention_team_plan(cu, [100, 100], 2, 7, 10, 100, 152,
                                            GB300_LIKE, 2)[0] == 0
    cu = np.array([0, 10, 20], np.int32)  # a prefix above the stated bound
    assert pb.pf_verify_attention_team_plan(cu, [100, 900], 2, 7, 10, 500, 152,
                                            GB300_LIKE, 2)[0] == 0
    assert pb.pf_verify_attention_team_plan(cu, [100, 100], 2, 0, 10, 100, 152,
                                            GB300_LIKE, 2)[0] == -1
    assert pb.pf_verify_attention_team_plan(cu, [100, 100], 2, 7, 10, 100, 0,
                                            GB300_LIKE, 2)[0] == -1


def test_null_pointers_and_the_device_figures():
    """NULL arrays are rejected; without a cluster-fit table the figures come
    from the current device, so without a GPU the call is refused."""
    import torch
    L = pb.lib()
    entries = np.zeros(pb.PF_TEAM_MAX_CTAS, np.uint32)
    out = np.zeros(3, np.int32)
    cu = np.array([0, 10, 20], np.int32)
    P = np.array([300, 900], np.int32)
    args = [cu.ctypes.data, P.ctypes.data, 2, 4, 7, 10, 900, 152, None, 2, entries.ctypes.data,
            out[0:].ctypes.data, out[1:].ctypes.data, out[2:].ctypes.data]
    for i in (0, 1, 10, 11, 12, 13):
        bad = list(args)
        bad[i] = None
        assert L.pf_verify_attention_team_plan(*bad) == -1
    st = L.pf_verify_attention_team_plan(*args)
    if torch.cuda.is_available():
        assert st in (0, 1)
    else:
        assert st == -1
