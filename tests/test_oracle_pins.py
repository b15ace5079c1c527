"""The fp64 oracle against its pins, and planted mistakes against the pins.

CPU only.  A planted mistake lives in a copy of an oracle function made
here; the oracle itself is never modified."""
import math

import numpy as np
import pytest

import oracle
from oracle import attention, accept, commit, lmhead, tree
from tests import oracle_checks as C


@pytest.mark.parametrize("check", C.ATTENTION_CHECKS, ids=lambda f: f.__name__)
def test_attention_pins(check):
    check(attention.tree_attention)


@pytest.mark.parametrize("check", C.LMHEAD_CHECKS, ids=lambda f: f.__name__)
def test_lmhead_pins(check):
    check(lmhead.logits, lmhead.greedy)


@pytest.mark.parametrize("check", C.ACCEPT_CHECKS, ids=lambda f: f.__name__)
def test_accept_pins(check):
    check(accept.accept_walk)


@pytest.mark.parametrize("check", C.COMMIT_CHECKS, ids=lambda f: f.__name__)
def test_commit_pins(check):
    check(commit.commit_rows)


def test_tree_pins():
    C.check_tree_structure(tree.validate, tree.depths, tree.ancestors_or_self)


# ----------------------------------------------------------------------------
# planted mistakes: each must be caught by at least one pin
# ----------------------------------------------------------------------------
def _attn_variant(visible_fn=None, kv_head=None, scale_fn=None, use_prefix=True):
    """A copy of the oracle's attention with one ingredient replaced."""
    def fn(q, pk, pv, tk, tv, parent, scale=None):
        q, pk, pv, tk, tv = (np.asarray(x, dtype=np.float64) for x in (q, pk, pv, tk, tv))
        N, Hq, D = q.shape
        Hkv = tk.shape[1]
        G = Hq // Hkv
        sc = (scale_fn or (lambda d: 1.0 / math.sqrt(d)))(D)
        out = np.zeros((N, Hq, D))
        for n in range(N):
            vis = sorted((visible_fn or tree.ancestors_or_self)(parent, n))
            for h in range(Hq):
                g = (kv_head or (lambda h, G, Hkv: h // G))(h, G, Hkv)
                keys = np.concatenate([pk[g] if use_prefix else pk[g][:0], tk[vis, g]], 0)
                vals = np.concatenate([pv[g] if use_prefix else pv[g][:0], tv[vis, g]], 0)
                s = keys @ q[n, h] * sc
                w = np.exp(s - s.max())
                out[n, h] = (w / w.sum()) @ vals
        return out
    return fn


ATTN_MUTANTS = {
    "drop_self": _attn_variant(visible_fn=lambda p, n: tree.ancestors_or_self(p, n) - {n}),
    "drop_root": _attn_variant(visible_fn=lambda p, n: tree.ancestors_or_self(p, n) - {0} or {n}),
    "no_tree_mask": _attn_variant(visible_fn=lambda p, n: set(range(len(p)))),
    "causal_by_index": _attn_variant(visible_fn=lambda p, n: set(range(n + 1))),
    "gqa_modulo": _attn_variant(kv_head=lambda h, G, Hkv: h % Hkv),
    "scale_one": _attn_variant(scale_fn=lambda d: 1.0),
    "scale_over_d": _attn_variant(scale_fn=lambda d: 1.0 / d),
    "drop_prefix": _attn_variant(use_prefix=False),
}


def _fails_some(checks, *impl):
    failed = 0
    for c in checks:
        try:
            c(*impl)
        except AssertionError:
            failed += 1
    return failed


@pytest.mark.parametrize("name", sorted(ATTN_MUTANTS))
def test_attention_mutants_caught(name):
    assert _fails_some(C.ATTENTION_CHECKS, ATTN_MUTANTS[name]) > 0


def _greedy_ties_high(lg):
    lg = np.asarray(lg, dtype=np.float64)
    am = lg.shape[1] - 1 - np.argmax(lg[:, ::-1], axis=1)
    top = lg[np.arange(len(lg)), am]
    rest = lg.copy()
    rest[np.arange(len(lg)), am] = -np.inf
    return am, top - rest.max(axis=1), top


def _greedy_margin_vs_min(lg):
    am, _, top = lmhead.greedy(lg)
    return am, top - np.asarray(lg).min(axis=1), top


def _logits_dropped_last_column(hidden, weight, chunk=8192):
    return np.asarray(hidden)[:, :-1] @ np.asarray(weight, dtype=np.float64)[:, :-1].T


def _logits_chunk_offset(hidden, weight, chunk=8192):
    """Off-by-one in the weight chunk loop: the first row of each chunk is skipped."""
    hidden = np.asarray(hidden, dtype=np.float64)
    V = weight.shape[0]
    out = np.zeros((hidden.shape[0], V))
    for s in range(0, V, chunk):
        e = min(V, s + chunk)
        out[:, s + 1:e] = hidden @ np.asarray(weight[s + 1:e], dtype=np.float64).T
    return out


LM_MUTANTS = {
    "ties_to_highest": (lmhead.logits, _greedy_ties_high),
    "margin_vs_min": (lmhead.logits, _greedy_margin_vs_min),
    "dropped_term": (_logits_dropped_last_column, lmhead.greedy),
    "chunk_off_by_one": (_logits_chunk_offset, lmhead.greedy),
}


@pytest.mark.parametrize("name", sorted(LM_MUTANTS))
def test_lmhead_mutants_caught(name):
    assert _fails_some(C.LMHEAD_CHECKS, *LM_MUTANTS[name]) > 0


def _walk_variant(no_bonus=False, highest_child=False, stop_early=False, bonus_of_parent=False):
    def fn(parent, tokens, greedy):
        n = len(parent)
        path = [0]
        while True:
            u = path[-1]
            order = range(n - 1, -1, -1) if highest_child else range(n)
            nxt = next((c for c in order if parent[c] == u and tokens[c] == greedy[u]), None)
            if nxt is None or (stop_early and len(path) >= 2):
                break
            path.append(nxt)
        a = len(path) - 1
        bonus_node = path[-2] if bonus_of_parent and len(path) > 1 else path[-1]
        out = [int(tokens[c]) for c in path[1:]]
        if not no_bonus:
            out.append(int(greedy[bonus_node]))
        return a, path, out, path[-1]
    return fn


WALK_MUTANTS = {
    "no_bonus": _walk_variant(no_bonus=True),
    "highest_child": _walk_variant(highest_child=True),
    "stop_after_one": _walk_variant(stop_early=True),
    "bonus_from_parent": _walk_variant(bonus_of_parent=True),
}


@pytest.mark.parametrize("name", sorted(WALK_MUTANTS))
def test_accept_mutants_caught(name):
    assert _fails_some(C.ACCEPT_CHECKS, WALK_MUTANTS[name]) > 0


def _commit_shifted(cache, P, path, tree_rows):
    out = np.array(cache, copy=True)
    for k, node in enumerate(path):
        out[:, P + k + 1 if P + k + 1 < out.shape[1] else P + k, :] = tree_rows[node]
    return out, P + len(path)


def _commit_drafts_only(cache, P, path, tree_rows):
    out = np.array(cache, copy=True)
    for k, node in enumerate(path[1:]):
        out[:, P + k, :] = tree_rows[node]
    return out, P + len(path) - 1


@pytest.mark.parametrize("mut", [_commit_shifted, _commit_drafts_only])
def test_commit_mutants_caught(mut):
    assert _fails_some(C.COMMIT_CHECKS, mut) > 0


def test_step_composes_the_parts():
    """The whole-step helper returns what its parts return."""
    rng = np.random.default_rng(11)
    N, P, Hq, Hkv, D, H, V, S = 4, 6, 2, 1, 8, 5, 13, 16
    parent = [-1, 0, 1, 1]
    layers = []
    for _ in range(2):
        L = dict(q=rng.standard_normal((N, Hq, D)), prefix_k=rng.standard_normal((Hkv, P, D)),
                 prefix_v=rng.standard_normal((Hkv, P, D)), tree_k=rng.standard_normal((N, Hkv, D)),
                 tree_v=rng.standard_normal((N, Hkv, D)))
        L["cache_k"] = np.zeros((Hkv, S, D))
        L["cache_v"] = np.zeros((Hkv, S, D))
        layers.append(L)
    hidden = rng.standard_normal((N, H))
    weight = rng.standard_normal((V, H))
    am = np.argmax(hidden @ weight.T, axis=1)
    tokens = [1, int(am[0]), int(am[1]), (int(am[1]) + 1) % V]
    r = oracle.step.verify_step(layers, hidden, weight, parent, tokens, P)
    assert r["accept_len"] == 2 and r["path"] == [0, 1, 2] and r["new_len"] == P + 3
    np.testing.assert_array_equal(r["caches"][1][0][:, P + 2], layers[1]["tree_k"][2])


# ----------------------------------------------------------------------------
# rotary re-rotation (rolling-image carryover)
# ----------------------------------------------------------------------------
from oracle import rope as R


@pytest.mark.parametrize("check", C.ROPE_CHECKS, ids=lambda f: f.__name__)
def test_rope_pins(check):
    check(R.carry_keys)


def test_rope_block_move_pin():
    C.check_rope_block_move(R.shift_block, R.carry_keys)


def _rope_variant(sign=1.0, interleaved=False, exponent=2.0, skip_inverse=False):
    def rotate(x, position, base):
        x = np.asarray(x, dtype=np.float64)
        D = x.shape[-1]
        ang = sign * position * base ** (-exponent * np.arange(D // 2) / D)
        c, s = np.cos(ang), np.sin(ang)
        if interleaved:
            x1, x2 = x[..., 0::2], x[..., 1::2]
            out = np.empty_like(x)
            out[..., 0::2] = x1 * c - x2 * s
            out[..., 1::2] = x1 * s + x2 * c
            return out
        x1, x2 = x[..., : D // 2], x[..., D // 2:]
        return np.concatenate([x1 * c - x2 * s, x1 * s + x2 * c], axis=-1)

    def carry(k, m, m_new, base):
        return rotate(k, m_new, base) if skip_inverse else rotate(rotate(k, -m, base), m_new, base)
    return carry


ROPE_MUTANTS = {
    "inverse_direction": _rope_variant(sign=-1.0),
    "interleaved_pairs": _rope_variant(interleaved=True),
    "wrong_frequency": _rope_variant(exponent=1.0),
    "no_inverse": _rope_variant(skip_inverse=True),
}


@pytest.mark.parametrize("name", sorted(ROPE_MUTANTS))
def test_rope_mutants_caught(name):
    assert _fails_some(C.ROPE_CHECKS, ROPE_MUTANTS[name]) > 0


def test_rope_block_mutants_caught():
    def values_rotated(K, V, src, dst, n, base):
        K2, V2 = R.shift_block(K, V, src, dst, n, base)
        for j in range(n):
            V2[:, dst + j] = R.carry_keys(V[:, src + j], src + j, dst + j, base)
        return K2, V2

    def reads_after_write(K, V, src, dst, n, base):
        K2 = np.array(K, dtype=np.float64, copy=True)
        V2 = np.array(V, dtype=np.float64, copy=True)
        for j in range(n):  # in-place without staging: overlapping sources get clobbered
            K2[:, dst + j] = R.carry_keys(K2[:, src + j], src + j, dst + j, base)
            V2[:, dst + j] = V2[:, src + j]
        return K2, V2
    for mut in (values_rotated, reads_after_write):
        with pytest.raises(AssertionError):
            C.check_rope_block_move(mut, R.carry_keys)


# ----------------------------------------------------------------------------
# decoding-memory retrieval
# ----------------------------------------------------------------------------
from oracle import retrieval as RV


@pytest.mark.parametrize("check", C.RETRIEVAL_CHECKS, ids=lambda f: f.__name__)
def test_retrieval_pins(check):
    check(RV.cosine_top1)


def test_project_key_pins():
    C.check_project_key(RV.project_key)


def _top1_variant(ties_high=False, no_boundary=False, no_token=False, raw_dot=False,
                  zero_is_orthogonal=False):
    def fn(qkey, keys, tok, pos, bound, y, lo=0, hi=None):
        hi = len(keys) if hi is None else hi
        q = np.asarray(qkey, dtype=np.float64)
        best, bestv = -1, None
        for j in range(lo, hi):
            if not no_token and int(tok[j]) != int(y):
                continue
            if not no_boundary and not int(pos[j]) < int(bound[j]):
                continue
            k = np.asarray(keys[j], dtype=np.float64)
            if not k.any():
                if not zero_is_orthogonal:
                    continue
                v = 0.0
            else:
                v = k @ q if raw_dot else (k @ q) / (np.linalg.norm(k) * np.linalg.norm(q))
            if best < 0 or v > bestv or (ties_high and v == bestv):
                best, bestv = j, v
        if best < 0:
            return -1, float("nan")
        k = np.asarray(keys[best], dtype=np.float64)
        if not k.any():
            return best, 0.0
        return best, float((k @ q) / (np.linalg.norm(k) * np.linalg.norm(q)))
    return fn


RETRIEVAL_MUTANTS = {
    "ties_to_highest": _top1_variant(ties_high=True),
    "ignores_boundary": _top1_variant(no_boundary=True),
    "ignores_token": _top1_variant(no_token=True),
    "raw_dot_product": _top1_variant(raw_dot=True),
    "zero_key_as_orthogonal": _top1_variant(zero_is_orthogonal=True),
}


@pytest.mark.parametrize("name", sorted(RETRIEVAL_MUTANTS))
def test_retrieval_mutants_caught(name):
    assert _fails_some(C.RETRIEVAL_CHECKS, RETRIEVAL_MUTANTS[name]) > 0


def test_project_key_mutants_caught():
    def round_half_up(h, proj):
        key, x = RV.project_key(h, proj)
        return np.floor(x + 0.5).astype(np.int8), x

    def no_normalise(h, proj):
        z = np.asarray(proj, dtype=np.float64) @ np.asarray(h, dtype=np.float64)
        x = np.clip(z, -127, 127)
        return np.rint(x).astype(np.int8), x
    for mut in (round_half_up, no_normalise):
        with pytest.raises(AssertionError):
            C.check_project_key(mut)


# ----------------------------------------------------------------------------
# prompt-prefix carryover
# ----------------------------------------------------------------------------
from oracle import prefix as PX


@pytest.mark.parametrize("check", C.PREFIX_CHECKS, ids=lambda f: f.__name__)
def test_prefix_pins(check):
    check(PX.common_prefix)


def test_prefix_carry_over():
    assert PX.carry_over([3, 4, 5, 6], [3, 4, 9, 6, 7]) == (2, 2, 3)


def _lcp_off_by_one(a, b):
    return min(PX.common_prefix(a, b) + 1, min(len(a), len(b)))


def _lcp_shorter_only(a, b):
    # forgets that a prompt ending early ends the common prefix
    p = PX.common_prefix(a, b)
    return max(p, min(len(a), len(b))) if p == 0 else p


def _lcp_last_mismatch(a, b):
    n = min(len(a), len(b))
    diff = [i for i in range(n) if int(a[i]) != int(b[i])]
    return diff[-1] if diff else n


@pytest.mark.parametrize("mut", [_lcp_off_by_one, _lcp_shorter_only, _lcp_last_mismatch])
def test_prefix_mutants_caught(mut):
    assert _fails_some(C.PREFIX_CHECKS, mut) > 0


# ----------------------------------------------------------------------------
# proposal-length controller (eq. 1)
# ----------------------------------------------------------------------------
from oracle import controller as CT


def test_controller_pins():
    C.check_expected_accepted_closed_forms(CT.expected_accepted)
    C.check_select_length_cases(CT.select_length)
    C.check_latency_fit_exact(CT.LatencyModel)
    C.check_acceptance_consistency(CT.AcceptanceModel)


def test_controller_mutants_caught():
    def no_plus_one(t, p1, pc, L):
        best, bo = 0, None
        for ell in range(L + 1):
            o = t[ell] / max(CT.expected_accepted(p1[ell], pc[ell], ell), 1e-300)
            if bo is None or o < bo:
                best, bo = ell, o
        return best, bo

    def ties_longest(t, p1, pc, L):
        best, bo = 0, None
        for ell in range(L + 1):
            o = t[ell] / (CT.expected_accepted(p1[ell], pc[ell], ell) + 1.0)
            if bo is None or o <= bo:
                best, bo = ell, o
        return best, bo

    for mut in (no_plus_one, ties_longest):
        assert _fails_some(C.CONTROLLER_CHECKS, mut) > 0

    def off_by_one_sum(p1, pc, ell):
        return sum(p1 * pc ** k for k in range(1, ell + 1))
    with pytest.raises(AssertionError):
        C.check_expected_accepted_closed_forms(off_by_one_sum)

    class LinearLatency(CT.LatencyModel):   # fits T, not log T
        def update(self, ell, t):
            super().update(ell, math.exp(t / 100.0))
    with pytest.raises(AssertionError):
        C.check_latency_fit_exact(LinearLatency)

    class NoContinuation(CT.AcceptanceModel):   # continuation trials dropped
        def update(self, ell, s, accepted):
            x = self._x(ell, s)
            self._step(self.w1, x, 1.0 if accepted >= 1 else 0.0, self.lr)
    with pytest.raises(AssertionError):
        C.check_acceptance_consistency(NoContinuation)
