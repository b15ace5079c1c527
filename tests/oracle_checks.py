"""Checks that pin the fp64 oracle to something other than itself.

Each ``check_*`` takes the implementation under test (normally the oracle's
own function) and raises AssertionError when it disagrees with a hand-derived
fixture, a library special case, an exact brute force or an invariant.  The
mutation tests hand these checks deliberately broken copies of the oracle
and require at least one check to fail, so a plausible slip (a dropped
term, a wrong index, a wrong sign) cannot pass unnoticed.
"""
import itertools
import math
import os

import numpy as np
import torch

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _nums(s):
    return [float(x) for x in s.split()]


def _rows(s):
    return np.array([_nums(r) for r in s.split("|")], dtype=np.float64)


def read_kv(name):
    out = {}
    for line in open(os.path.join(GOLDEN, name)):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        k, v = line.split(":", 1)
        out[k.strip()] = v.strip()
    return out


# ----------------------------------------------------------------------------
# attention
# ----------------------------------------------------------------------------
def _sdpa(q, k, v, mask, scale):
    """torch's scaled_dot_product_attention in float64 on the CPU:
    q [Hq, M, D], k/v [Hq, S, D], mask [M, S] bool (True = attend)."""
    with torch.no_grad():
        o = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q)[None], torch.from_numpy(k)[None],
            torch.from_numpy(v)[None], attn_mask=torch.from_numpy(mask),
            scale=scale)
    return o[0].numpy()


def _expand_gqa(x, G):
    """[Hkv, S, D] -> [Hkv*G, S, D], query head h uses KV head h // G."""
    return np.repeat(x, G, axis=0)


def _random_attention_case(rng, N, P, Hq, Hkv, D, parent):
    q = rng.standard_normal((N, Hq, D))
    pk = rng.standard_normal((Hkv, P, D))
    pv = rng.standard_normal((Hkv, P, D))
    tk = rng.standard_normal((N, Hkv, D))
    tv = rng.standard_normal((N, Hkv, D))
    return q, pk, pv, tk, tv, np.asarray(parent)


def check_attention_golden(attn):
    g = read_kv("attention_worked.txt")
    parent = np.array(_nums(g["parent"]), dtype=np.int64)
    N = len(parent)
    q = np.tile(np.array(_nums(g["q"]))[None, None, :], (N, 1, 1))
    pk = np.array(_nums(g["prefix_k"]))[None, None, :]
    pv = np.array(_nums(g["prefix_v"]))[None, None, :]
    tk = _rows(g["tree_k"])[:, None, :]
    tv = _rows(g["tree_v"])[:, None, :]
    out = attn(q, pk, pv, tk, tv, parent)
    for n in range(N):
        np.testing.assert_allclose(out[n, 0], _nums(g[f"out{n}"]), rtol=0, atol=1e-12)


def check_attention_chain_is_causal(attn, seed=1):
    """A linear chain is ordinary causal attention over prefix + chain."""
    rng = np.random.default_rng(seed)
    N, P, Hq, Hkv, D = 7, 11, 4, 2, 8
    parent = np.arange(-1, N - 1)
    q, pk, pv, tk, tv, parent = _random_attention_case(rng, N, P, Hq, Hkv, D, parent)
    K = np.concatenate([pk, tk.transpose(1, 0, 2)], axis=1)
    V = np.concatenate([pv, tv.transpose(1, 0, 2)], axis=1)
    G = Hq // Hkv
    mask = np.arange(P + N)[None, :] <= (P + np.arange(N))[:, None]
    ref = _sdpa(q.transpose(1, 0, 2), _expand_gqa(K, G), _expand_gqa(V, G), mask,
                1.0 / math.sqrt(D))
    np.testing.assert_allclose(attn(q, pk, pv, tk, tv, parent), ref.transpose(1, 0, 2),
                               rtol=0, atol=1e-10)


def _children(parent):
    ch = {i: [] for i in range(len(parent))}
    for j in range(1, len(parent)):
        ch[int(parent[j])].append(j)
    return ch


def _paths_by_dfs(parent):
    """Every root -> node path, found by depth-first search over child lists."""
    ch = _children(parent)
    paths = {}
    stack = [[0]]
    while stack:
        p = stack.pop()
        paths[p[-1]] = p
        for c in ch[p[-1]]:
            stack.append(p + [c])
    return paths


def check_attention_tree_paths(attn, seed=2):
    """Brute force: node n of a tree equals the last query of plain attention
    over prefix + its own root path (one SDPA call per node)."""
    rng = np.random.default_rng(seed)
    N, P, Hq, Hkv, D = 10, 5, 6, 2, 8
    parent = [-1, 0, 0, 1, 1, 2, 4, 4, 3, 6]
    q, pk, pv, tk, tv, parent = _random_attention_case(rng, N, P, Hq, Hkv, D, parent)
    out = attn(q, pk, pv, tk, tv, parent)
    G = Hq // Hkv
    for n, path in _paths_by_dfs(parent).items():
        K = np.concatenate([pk, tk[path].transpose(1, 0, 2)], axis=1)
        V = np.concatenate([pv, tv[path].transpose(1, 0, 2)], axis=1)
        mask = np.ones((1, K.shape[1]), dtype=bool)
        ref = _sdpa(q[n][:, None, :], _expand_gqa(K, G), _expand_gqa(V, G), mask,
                    1.0 / math.sqrt(D))
        np.testing.assert_allclose(out[n], ref[:, 0, :], rtol=0, atol=1e-10)


def check_attention_star_and_root(attn, seed=3):
    """Star tree = independent single-query decodes; N = 1 = plain decode;
    P = 0 = attention over the node's own path only."""
    rng = np.random.default_rng(seed)
    Hq, Hkv, D = 4, 1, 16
    for N, P in ((6, 9), (1, 13), (5, 0)):
        parent = [-1] + [0] * (N - 1)
        q, pk, pv, tk, tv, parent = _random_attention_case(rng, N, P, Hq, Hkv, D, parent)
        out = attn(q, pk, pv, tk, tv, parent)
        for n in range(N):
            rows = [0] if n == 0 else [0, n]
            K = np.concatenate([pk, tk[rows].transpose(1, 0, 2)], axis=1)
            V = np.concatenate([pv, tv[rows].transpose(1, 0, 2)], axis=1)
            ref = _sdpa(q[n][:, None, :], _expand_gqa(K, Hq), _expand_gqa(V, Hq),
                        np.ones((1, K.shape[1]), dtype=bool), 1.0 / math.sqrt(D))
            np.testing.assert_allclose(out[n], ref[:, 0, :], rtol=0, atol=1e-10)


def check_attention_uniform_values(attn, seed=4):
    """If every visible value row equals c, the output is c whatever the scores."""
    rng = np.random.default_rng(seed)
    N, P, Hq, Hkv, D = 5, 7, 4, 2, 8
    parent = [-1, 0, 1, 1, 0]
    q, pk, _, tk, _, parent = _random_attention_case(rng, N, P, Hq, Hkv, D, parent)
    c = rng.standard_normal((Hkv, D))
    pv = np.repeat(c[:, None, :], P, axis=1)
    tv = np.repeat(c[None, :, :], N, axis=0)
    out = attn(q * 3.0, pk, pv, tk, tv, parent)
    for h in range(Hq):
        np.testing.assert_allclose(out[:, h, :], np.repeat(c[h // (Hq // Hkv)][None], N, 0),
                                   rtol=0, atol=1e-12)


ATTENTION_CHECKS = [check_attention_golden, check_attention_chain_is_causal,
                    check_attention_tree_paths, check_attention_star_and_root,
                    check_attention_uniform_values]


# ----------------------------------------------------------------------------
# LM head and greedy prediction
# ----------------------------------------------------------------------------
def check_lmhead_golden(logits_fn, greedy_fn):
    g = read_kv("lmhead_worked.txt")
    hidden, weight = _rows(g["hidden"]), _rows(g["weight"])
    lg = logits_fn(hidden, weight)
    np.testing.assert_array_equal(lg[0], _nums(g["logits0"]))
    np.testing.assert_array_equal(lg[1], _nums(g["logits1"]))
    am, margin, _ = greedy_fn(lg)
    np.testing.assert_array_equal(am, [int(x) for x in _nums(g["argmax"])])
    np.testing.assert_array_equal(margin, _nums(g["margin"]))


def check_lmhead_exact_integers(logits_fn, greedy_fn, seed=5):
    """Small-integer inputs: every logit is exact, so compare with Python
    integer dot products, and argmax/margin with a scan written out here."""
    rng = np.random.default_rng(seed)
    N, V, H = 5, 37, 23
    hidden = rng.integers(-3, 4, size=(N, H))
    weight = rng.integers(-3, 4, size=(V, H))
    lg = logits_fn(hidden.astype(np.float64), weight.astype(np.float64), chunk=8)
    for n in range(N):
        row = [sum(int(hidden[n, c]) * int(weight[v, c]) for c in range(H)) for v in range(V)]
        assert list(lg[n].astype(np.int64)) == row
        best = max(row)
        first = row.index(best)
        second = max(x for i, x in enumerate(row) if i != first)
        am, margin, top = greedy_fn(lg[n:n + 1])
        assert int(am[0]) == first and margin[0] == best - second and top[0] == best


def check_lmhead_ties_lowest(logits_fn, greedy_fn):
    lg = np.array([[0.5, 2.0, 2.0, -1.0], [3.0, 3.0, 3.0, 3.0], [-2.0, -1.0, -3.0, -1.0]])
    am, margin, _ = greedy_fn(lg)
    assert list(am) == [1, 0, 1]
    assert list(margin) == [0.0, 0.0, 0.0]


def check_lmhead_float_bruteforce(logits_fn, greedy_fn, seed=6):
    """Random float64 inputs against math.fsum dot products."""
    rng = np.random.default_rng(seed)
    hidden = rng.standard_normal((3, 19))
    weight = rng.standard_normal((29, 19))
    lg = logits_fn(hidden, weight, chunk=7)
    for n in range(3):
        for v in range(29):
            ref = math.fsum(float(hidden[n, c]) * float(weight[v, c]) for c in range(19))
            assert abs(lg[n, v] - ref) <= 1e-12 * (1 + abs(ref))


LMHEAD_CHECKS = [check_lmhead_golden, check_lmhead_exact_integers,
                 check_lmhead_ties_lowest, check_lmhead_float_bruteforce]


# ----------------------------------------------------------------------------
# acceptance
# ----------------------------------------------------------------------------
def _ints(s):
    return [int(x) for x in s.split()]


def check_accept_golden(walk):
    for line in open(os.path.join(GOLDEN, "accept_worked.txt")):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        lhs, rhs = line.split("||")
        parent, tokens, greedy = [_ints(x) for x in lhs.split("|")]
        a, path, out_tokens, last = [x.strip() for x in rhs.split("|")]
        got = walk(parent, tokens, greedy)
        assert got[0] == int(a), (line, got)
        assert list(got[1]) == _ints(path), (line, got)
        assert list(got[2]) == _ints(out_tokens), (line, got)
        assert got[3] == int(last), (line, got)


def check_accept_chain_prefix(walk, seed=7):
    """Chain: accepted length = longest draft prefix equal to the greedy
    predictions (Section 3.2), for every planted length."""
    rng = np.random.default_rng(seed)
    for ell in (0, 1, 2, 5, 12):
        for planted in range(ell + 1):
            greedy = rng.integers(0, 50, size=ell + 1)
            drafts = [int(greedy[i]) if i < planted else int((greedy[i] + 1 + rng.integers(48)) % 50)
                      for i in range(ell)]
            tokens = [int(rng.integers(50))] + drafts
            parent = list(range(-1, ell))
            a, path, out_tokens, last = walk(parent, tokens, greedy)
            assert a == planted
            assert list(path) == list(range(planted + 1))
            assert list(out_tokens) == drafts[:planted] + [int(greedy[planted])]
            assert last == planted


def check_accept_exhaustive(walk, seed=8):
    """Trees with distinct sibling tokens: the walk's path is the unique
    longest root path whose every edge matches the parent's prediction,
    found by enumerating all node subsets that form root paths."""
    rng = np.random.default_rng(seed)
    for trial in range(60):
        N = int(rng.integers(1, 9))
        parent = [-1] + [int(rng.integers(0, j)) for j in range(1, N)]
        V = 6
        greedy = rng.integers(0, V, size=N)
        tokens = [int(rng.integers(V))]
        used = {}
        for j in range(1, N):
            choices = [t for t in range(V) if t not in used.get(parent[j], set())]
            t = int(choices[rng.integers(len(choices))])
            used.setdefault(parent[j], set()).add(t)
            tokens.append(t)
        best = [0]
        for r in range(1, N + 1):
            for subset in itertools.combinations(range(N), r):
                if subset[0] != 0:
                    continue
                ok = all(parent[subset[i]] == subset[i - 1] and
                         tokens[subset[i]] == greedy[subset[i - 1]] for i in range(1, r))
                if ok and r > len(best):
                    best = list(subset)
        a, path, out_tokens, last = walk(parent, tokens, greedy)
        assert list(path) == best, (parent, tokens, list(greedy), path, best)
        assert a == len(best) - 1 and last == best[-1]
        assert list(out_tokens) == [tokens[c] for c in best[1:]] + [int(greedy[best[-1]])]


ACCEPT_CHECKS = [check_accept_golden, check_accept_chain_prefix, check_accept_exhaustive]


# ----------------------------------------------------------------------------
# commit
# ----------------------------------------------------------------------------
def check_commit_postcondition(commit, seed=9):
    """Rows P..P+a hold the accepted path's tree rows; every other cache row
    is untouched; the new length is P + a + 1."""
    rng = np.random.default_rng(seed)
    Hkv, S, D, N = 2, 20, 4, 6
    for P, path in ((5, [0, 2, 3]), (0, [0]), (14, [0, 1, 4, 5])):
        cache = rng.standard_normal((Hkv, S, D))
        tree = rng.standard_normal((N, Hkv, D))
        new, n1 = commit(cache, P, path, tree)
        assert n1 == P + len(path)
        for pos in range(S):
            if P <= pos < P + len(path):
                np.testing.assert_array_equal(new[:, pos, :], tree[path[pos - P]])
            else:
                np.testing.assert_array_equal(new[:, pos, :], cache[:, pos, :])


COMMIT_CHECKS = [check_commit_postcondition]


# ----------------------------------------------------------------------------
# tree structure
# ----------------------------------------------------------------------------
def check_tree_structure(validate, depths, ancestors):
    assert validate([-1]) and validate([-1, 0, 0, 1, 2])
    for bad in ([], [0], [-1, 1], [-1, 0, 2], [-1, -1], [-1, 0, 3, 1]):
        assert not validate(bad), bad
    parent = [-1, 0, 0, 1, 3, 2]
    assert list(depths(parent)) == [0, 1, 1, 2, 3, 2]
    assert ancestors(parent, 4) == {0, 1, 3, 4}
    assert ancestors(parent, 5) == {0, 2, 5}
    assert ancestors(parent, 0) == {0}



# ----------------------------------------------------------------------------
# rotary re-rotation (rolling-image carryover)
# ----------------------------------------------------------------------------
def _complex_rope(x, position, base):
    """Rotary embedding written as complex multiplication: pair i is the
    complex number x_i + 1j * x_{i+D/2}, turned by exp(1j * position * theta_i)."""
    x = np.asarray(x, dtype=np.float64)
    D = x.shape[-1]
    theta = np.array([base ** (-(2.0 * i) / D) for i in range(D // 2)])
    z = (x[..., : D // 2] + 1j * x[..., D // 2:]) * np.exp(1j * position * theta)
    return np.concatenate([z.real, z.imag], axis=-1)


def check_rope_golden(carry):
    g = read_kv("rope_worked.txt")
    out = carry(np.array(_nums(g["key"])), float(g["m"]), float(g["m_new"]), float(g["base"]))
    np.testing.assert_allclose(out, _nums(g["expect"]), rtol=0, atol=1e-9)


def check_rope_carry_is_relative(carry, seed=10):
    """Carrying a key rotated at m to m' equals embedding the raw key at m'
    (complex-multiplication form), for several shifts, both directions."""
    rng = np.random.default_rng(seed)
    for D, base in ((8, 10000.0), (64, 1e6), (128, 1e6)):
        k = rng.standard_normal((3, D))
        for m, m_new in ((0, 7), (1300, 17), (5, 4096), (123, 123)):
            got = carry(_complex_rope(k, m, base), m, m_new, base)
            np.testing.assert_allclose(got, _complex_rope(k, m_new, base), rtol=0, atol=1e-9)
            np.testing.assert_allclose(np.linalg.norm(got, axis=-1), np.linalg.norm(k, axis=-1),
                                       rtol=1e-12)


def check_rope_block_move(shift, carry, seed=11):
    """shift_block: destination rows hold the re-rotated keys and the copied
    values; every other row keeps its contents; left and right moves, with
    and without overlap."""
    rng = np.random.default_rng(seed)
    Hkv, S, D, base = 2, 40, 8, 10000.0
    for src, dst, n in ((20, 5, 10), (5, 9, 12), (30, 2, 6), (0, 0, 4)):
        K = rng.standard_normal((Hkv, S, D))
        V = rng.standard_normal((Hkv, S, D))
        K2, V2 = shift(K, V, src, dst, n, base)
        for pos in range(S):
            if dst <= pos < dst + n:
                j = pos - dst
                np.testing.assert_allclose(K2[:, pos], carry(K[:, src + j], src + j, pos, base),
                                           rtol=0, atol=1e-12)
                np.testing.assert_array_equal(V2[:, pos], V[:, src + j])
            else:
                np.testing.assert_array_equal(K2[:, pos], K[:, pos])
                np.testing.assert_array_equal(V2[:, pos], V[:, pos])


ROPE_CHECKS = [check_rope_golden, check_rope_carry_is_relative]


# ----------------------------------------------------------------------------
# decoding-memory retrieval
# ----------------------------------------------------------------------------
def _ints_rows(s):
    return np.array([[int(x) for x in r.split()] for r in s.split("|")], dtype=np.int8)


def check_retrieval_golden(top1):
    g = read_kv("retrieval_worked.txt")
    q = np.array([int(x) for x in g["q"].split()], dtype=np.int8)
    best, sim = top1(q, _ints_rows(g["keys"]), _ints(g["entry_token"]), _ints(g["entry_pos"]),
                     _ints(g["entry_bound"]), int(g["token"]))
    assert best == int(g["best"]) and abs(sim - float(g["similarity"])) < 1e-12


def check_retrieval_float_bruteforce(top1, seed=12):
    """Random int8 keys without near ties: the exact selection equals numpy's
    float64 cosine argmax over the eligible entries."""
    rng = np.random.default_rng(seed)
    for trial in range(20):
        M, D = 200, 32
        keys = rng.integers(-127, 128, size=(M, D)).astype(np.int8)
        q = rng.integers(-127, 128, size=D).astype(np.int8)
        tok = rng.integers(0, 4, size=M)
        pos = rng.integers(0, 10, size=M)
        bound = rng.integers(0, 10, size=M)
        y = int(rng.integers(0, 4))
        kf = keys.astype(np.float64)
        cos = kf @ q.astype(np.float64) / (np.linalg.norm(kf, axis=1) * np.linalg.norm(q))
        elig = (tok == y) & (pos < bound)
        best, sim = top1(q, keys, tok, pos, bound, y)
        if not elig.any():
            assert best == -1
            continue
        c = np.where(elig, cos, -np.inf)
        order = np.sort(c[elig])
        if len(order) > 1 and order[-1] - order[-2] < 1e-9:
            continue
        assert best == int(np.argmax(c)) and abs(sim - c.max()) < 1e-12


def check_retrieval_ties_and_ranges(top1):
    q = np.array([5, -3, 2, 0], dtype=np.int8)
    base = np.array([2, -1, 1, 0], dtype=np.int8)
    keys = np.stack([base * 3, base, base * 2, -base, base * 3]).astype(np.int8)
    tok = [1, 1, 1, 1, 1]
    pos = [0, 0, 0, 0, 0]
    bound = [1, 1, 1, 1, 1]
    assert top1(q, keys, tok, pos, bound, 1)[0] == 0          # equal cosines: lowest index
    assert top1(q, keys, tok, pos, bound, 1, lo=1)[0] == 1
    assert top1(q, keys, tok, pos, bound, 1, lo=3, hi=4)[0] == 3  # only a negative cosine left
    assert top1(q, keys, tok, pos, bound, 2)[0] == -1         # no entry with the token
    assert top1(q, keys, tok, pos, [0, 0, 0, 0, 0], 1)[0] == -1  # every entry at its boundary


def check_project_key(project):
    rng = np.random.default_rng(13)
    H = 96
    proj = rng.standard_normal((256, H))
    for _ in range(5):
        h = rng.standard_normal(H)
        key, x = project(h, proj)
        assert key.dtype == np.int8 and key.shape == (256,)
        assert np.abs(key).max() == 127
        assert np.array_equal(project(3.5 * h, proj)[0], key)   # scale of h is irrelevant
        z = proj @ (h / np.linalg.norm(h))
        assert np.dot(key, z) / (np.linalg.norm(key.astype(float)) * np.linalg.norm(z)) > 0.999
        assert np.all(np.abs(x - key) <= 0.5)
    # half-way values round to even
    proj2 = np.zeros((256, 4))
    proj2[0, 0] = 254.0       # -> 127 (the maximum)
    proj2[1, 0] = 5.0         # 127 * 5 / 254 = 2.5 -> 2
    proj2[2, 0] = 7.0         # 3.5 -> 4
    proj2[3, 0] = -3.0        # -1.5 -> -2
    key, _ = project(np.array([1.0, 0, 0, 0]), proj2)
    assert list(key[:4]) == [127, 2, 4, -2]


def check_retrieval_zero_keys(top1):
    """An all-zero key has no cosine: it is never selected, not even over
    entries of negative cosine, and alone it leaves nothing to select."""
    q = np.array([3, 1, -2, 4], dtype=np.int8)
    keys = np.array([[0, 0, 0, 0], [-3, -1, 2, -4], [0, 0, 0, 0]], dtype=np.int8)
    tok, pos, bound = [9, 9, 9], [0, 0, 0], [1, 1, 1]
    assert top1(q, keys, tok, pos, bound, 9)[0] == 1
    assert top1(q, keys, tok, pos, bound, 9, lo=2)[0] == -1
    assert top1(q, keys, tok, pos, bound, 9, hi=1)[0] == -1


RETRIEVAL_CHECKS = [check_retrieval_golden, check_retrieval_float_bruteforce,
                    check_retrieval_ties_and_ranges, check_retrieval_zero_keys]


# ----------------------------------------------------------------------------
# prompt-prefix carryover
# ----------------------------------------------------------------------------
def check_prefix_special_cases(lcp):
    assert lcp([], []) == 0
    assert lcp([5, 6, 7], []) == 0
    assert lcp([5, 6, 7], [5, 6, 7]) == 3              # identical prompts
    assert lcp([5, 6, 7], [5, 6, 7, 8, 9]) == 3        # the old prompt is a prefix
    assert lcp([5, 6, 7, 8, 9], [5, 6]) == 2           # the new prompt is a prefix
    assert lcp([1, 2, 3], [9, 2, 3]) == 0              # differs at the first token
    assert lcp([1, 2, 3, 4], [1, 2, 3, 5]) == 3        # differs at the last token
    assert lcp([-1, 0, 2**31 - 1], [-1, 0, 2**31 - 1]) == 3   # negative / extreme keys


def check_prefix_planted(lcp, seed=14):
    """A mismatch planted at position k of otherwise equal random prompts is
    found at k, in either argument order, whatever follows it."""
    rng = np.random.default_rng(seed)
    for _ in range(200):
        n = int(rng.integers(1, 300))
        a = rng.integers(0, 50, size=n)
        b = a.copy()
        k = int(rng.integers(0, n))
        b[k] = a[k] + 1 + int(rng.integers(0, 5))
        b[k + 1:] = rng.integers(0, 50, size=n - k - 1)   # anything may follow
        tail = rng.integers(0, 50, size=int(rng.integers(0, 20)))
        b = np.concatenate([b, tail])
        assert lcp(a, b) == k and lcp(b, a) == k


PREFIX_CHECKS = [check_prefix_special_cases, check_prefix_planted]


# ----------------------------------------------------------------------------
# proposal-length controller (eq. 1)
# ----------------------------------------------------------------------------
def check_expected_accepted_closed_forms(expected):
    for p1 in (0.0, 0.3, 1.0):
        assert expected(p1, 0.5, 0) == 0.0                       # no proposal, nothing accepted
        assert abs(expected(p1, 0.0, 7) - p1) < 1e-12            # never continues
        assert abs(expected(p1, 1.0, 7) - 7 * p1) < 1e-12        # always continues
    for pc in (0.2, 0.9):                                        # geometric series
        for ell in (1, 5, 64):
            assert abs(expected(0.7, pc, ell) - 0.7 * (1 - pc ** ell) / (1 - pc)) < 1e-12


def check_select_length_cases(select):
    L = 8
    # free verification, certain acceptance: the longest proposal
    assert select([1.0] * (L + 1), [1.0] * (L + 1), [1.0] * (L + 1), L)[0] == L
    # latency proportional to tokens produced: every length ties -> shortest
    assert select([1.0 + l for l in range(L + 1)], [1.0] * (L + 1), [1.0] * (L + 1), L)[0] == 0
    # nothing is ever accepted: greedy (l = 0) is cheapest
    assert select([1.0 + 0.1 * l for l in range(L + 1)], [0.0] * (L + 1), [0.5] * (L + 1), L)[0] == 0
    # hand-worked: T = (1, 1.2, 1.6), p1 = 0.5, pc = 0.5 -> objectives 1, 0.8, 0.91..
    best, obj = select([1.0, 1.2, 1.6], [0.5] * 3, [0.5] * 3, 2)
    assert best == 1 and abs(obj - 0.8) < 1e-12


def check_latency_fit_exact(model_cls):
    """Noise-free log-quadratic data are fitted exactly."""
    c = (5.5, 0.004, -8e-6)
    m = model_cls()
    for ell in (0, 1, 4, 16, 64, 127, 3, 32):
        m.update(ell, math.exp(c[0] + c[1] * ell + c[2] * ell * ell))
    for ell in (0, 10, 100):
        want = math.exp(c[0] + c[1] * ell + c[2] * ell * ell)
        assert abs(m.predict(ell) / want - 1.0) < 1e-6


def check_acceptance_consistency(model_cls, seed=15):
    """Bernoulli acceptance at fixed rates: the online estimates approach
    the rates (first token 0.8, continuation 0.6) at the trained (l, s)."""
    rng = np.random.default_rng(seed)
    m = model_cls(16, 0.05)
    for _ in range(6000):
        a = 0
        if rng.random() < 0.8:
            a = 1
            while a < 16 and rng.random() < 0.6:
                a += 1
        m.update(16, 0.9, a)
    p1, pc = m.predict(16, 0.9)
    assert abs(p1 - 0.8) < 0.05 and abs(pc - 0.6) < 0.05


CONTROLLER_CHECKS = [check_select_length_cases]
