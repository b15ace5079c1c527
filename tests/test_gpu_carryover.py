"""Rolling-image key re-rotation (Section 3.4) and decoding-memory retrieval
(Section 3.2, Section 4) through the C ABI against the fp64 oracle.

Tolerances.  pf_kv_shift computes each rotated pair in fp32 from fp32
cos/sin (rounded from double) and rounds once to the storage type, so a key
element differs from the fp64 result by at most half a unit in the last
place of the stored type (<= 2^-8 |x| for bf16, 2^-24 |x| for fp32) plus a
few fp32 roundings of the pair's magnitude; values and every row outside
the destination span are bit-exact.  pf_retrieve is exact (integer dot
products, exact comparison): the index is bit-exact and the similarity
within 1e-6.  pf_retrieval_key accumulates z in fp32: codes equal the
oracle's except where the oracle's pre-rounding value lies within 0.01 of a
rounding boundary, where they may differ by one."""
import ctypes as C

import numpy as np
import pytest
import torch

from oracle import retrieval as ORt
from oracle import rope as OR
from paper_2609_32166_gb300 import binding as pb
from paper_2609_32166_gb300 import inputs as I

pytestmark = pytest.mark.gpu


def _stream():
    return torch.cuda.current_stream().cuda_stream


def _dev(a: np.ndarray) -> torch.Tensor:
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def _host(t: torch.Tensor, like: np.ndarray) -> np.ndarray:
    out = t.cpu().numpy()
    return out.view(like.dtype) if like.dtype == np.uint16 else out


# ---------------------------------------------------------------------------
# pf_kv_shift
# ---------------------------------------------------------------------------
class ShiftCase:
    def __init__(self, dtype, layout, L, B, Hkv, D, S, seq, seed=0):
        self.dtype, self.layout, self.L, self.B, self.Hkv, self.D, self.S = (
            dtype, layout, L, B, Hkv, D, S)
        self.seq = seq
        if layout == "paged":
            self.pages_per_seq = -(-S // I.PAGE_SIZE)
            self.pt, self.num_pages = I.page_table(B, self.pages_per_seq, seed)
            shape = (L, self.num_pages, Hkv, I.PAGE_SIZE, D)
        else:
            shape = (L, B, Hkv, S, D)
        self.k0 = I.normal(shape, 1.0, seed, "shift_k", 0, dtype)
        self.v0 = I.normal(shape, 1.0, seed, "shift_v", 0, dtype)
        self.k = _dev(self.k0)
        self.v = _dev(self.v0)
        self.err = torch.zeros(1, dtype=torch.int32, device="cuda")
        if layout == "paged":
            self.pt_dev = _dev(self.pt)

    def desc(self, src, dst, count, base):
        d = pb.pf_shift_desc()
        d.dtype = pb.PF_BF16 if self.dtype == "bf16" else pb.PF_F32
        d.n_layers, d.n_kv_heads, d.head_dim = self.L, self.Hkv, self.D
        d.seq, d.batch, d.src, d.dst, d.count, d.rope_base = self.seq, self.B, src, dst, count, base
        d.cache.k, d.cache.v = self.k.data_ptr(), self.v.data_ptr()
        per_layer = int(np.prod(self.k0.shape[1:]))
        d.cache_layer_stride = per_layer
        if self.layout == "paged":
            d.cache.layout = pb.PF_KV_PAGED
            d.cache.page_table = self.pt_dev.data_ptr()
            d.cache.num_pages = self.num_pages
            d.cache.pages_per_seq = self.pages_per_seq
        else:
            d.cache.layout = pb.PF_KV_CONTIGUOUS
            d.cache.max_seq = self.S
        d.error_flag = self.err.data_ptr()
        return d

    def phys(self, pos):
        """(index tuple prefix) of logical position pos of the moved sequence."""
        if self.layout == "paged":
            return int(self.pt[self.seq, pos // I.PAGE_SIZE]), pos % I.PAGE_SIZE
        return self.seq, pos

    def logical_rows(self, arr, l):
        """[Hkv, S, D] rows of the moved sequence in layer l."""
        if self.layout == "paged":
            out = np.empty((self.Hkv, self.S, self.D), dtype=arr.dtype)
            for p in range(self.S):
                pg, r = self.phys(p)
                out[:, p, :] = arr[l, pg, :, r, :]
            return out
        return arr[l, self.seq]

    def run_and_check(self, src, dst, count, base):
        pb.pf_kv_shift(self.desc(src, dst, count, base), _stream())
        torch.cuda.synchronize()
        assert int(self.err.item()) == 0
        k1, v1 = _host(self.k, self.k0), _host(self.v, self.v0)
        moved = np.zeros(self.k0.shape[:-1], dtype=bool)
        for p in range(dst, dst + count):
            idx = self.phys(p)
            moved[(slice(None), idx[0], slice(None), idx[1])] = True
        # rows outside the destination span, in every layer, sequence and page
        assert np.array_equal(k1[~moved], self.k0[~moved])
        assert np.array_equal(v1[~moved], self.v0[~moved])
        D = self.D
        for l in range(self.L):
            K0 = I.as_f64(self.logical_rows(self.k0, l), self.dtype)
            V0 = I.as_f64(self.logical_rows(self.v0, l), self.dtype)
            Ko, Vo = OR.shift_block(K0, V0, src, dst, count, base)
            got_k = I.as_f64(self.logical_rows(k1, l), self.dtype)[:, dst:dst + count]
            got_v = self.logical_rows(v1, l)[:, dst:dst + count]
            assert np.array_equal(got_v, self.logical_rows(self.v0, l)[:, src:src + count])
            want = Ko[:, dst:dst + count]
            x = K0[:, src:src + count]
            pair = np.abs(x[..., : D // 2]) + np.abs(x[..., D // 2:])
            pair = np.concatenate([pair, pair], axis=-1)
            ulp_half = 2.0 ** -8 if self.dtype == "bf16" else 2.0 ** -24
            tol = ulp_half * np.abs(want) + 2.0 ** -20 * pair
            bad = np.abs(got_k - want) > tol
            assert not bad.any(), (l, np.argwhere(bad)[:5], got_k[bad][:5], want[bad][:5])


SHIFT_CASES = {
    # disjoint spans, several passes per segment
    "bf16-disjoint-left": dict(dtype="bf16", layout="contiguous", L=2, B=2, Hkv=2, D=128, S=1200,
                               seq=1, src=700, dst=100, count=450, base=1e4),
    # overlapping move to lower positions: 3 ascending segments of 260 rows
    "bf16-overlap-left": dict(dtype="bf16", layout="contiguous", L=2, B=1, Hkv=2, D=128, S=1100,
                              seq=0, src=300, dst=40, count=700, base=1e6),
    # overlapping move to higher positions, paged: 3 descending segments
    "bf16-paged-overlap-right": dict(dtype="bf16", layout="paged", L=2, B=3, Hkv=2, D=128,
                                     S=930, seq=2, src=50, dst=310, count=600, base=1e4),
    # shift of 5 rows over 500: one CTA per (layer, head) walks the passes in order
    "bf16-small-shift-left": dict(dtype="bf16", layout="contiguous", L=1, B=1, Hkv=3, D=128,
                                  S=600, seq=0, src=37, dst=32, count=500, base=1e4),
    "bf16-small-shift-right-paged": dict(dtype="bf16", layout="paged", L=1, B=2, Hkv=2, D=64,
                                         S=700, seq=0, src=3, dst=10, count=640, base=1e4),
    # fp32, D = 64, a single row
    "f32-one-row": dict(dtype="f32", layout="contiguous", L=3, B=1, Hkv=1, D=64, S=64, seq=0,
                        src=63, dst=0, count=1, base=1e4),
    # D = 48: three 16-byte chunks per half row, a pass ends mid-block
    "bf16-d48-ragged": dict(dtype="bf16", layout="contiguous", L=1, B=1, Hkv=2, D=48, S=900,
                            seq=0, src=17, dst=0, count=800, base=1e4),
    # D = 256 and angles up to 3e4 rad
    "bf16-d256-far": dict(dtype="bf16", layout="contiguous", L=1, B=1, Hkv=1, D=256, S=33000,
                          seq=0, src=0, dst=30000, count=2000, base=1e6),
    "f32-paged-d128": dict(dtype="f32", layout="paged", L=2, B=2, Hkv=2, D=128, S=400, seq=1,
                           src=200, dst=8, count=190, base=5e5),
}


@pytest.mark.parametrize("name", sorted(SHIFT_CASES))
def test_kv_shift_matches_oracle(name):
    c = dict(SHIFT_CASES[name])
    src, dst, count, base = c.pop("src"), c.pop("dst"), c.pop("count"), c.pop("base")
    ShiftCase(**c).run_and_check(src, dst, count, base)


def test_kv_shift_there_and_back():
    """Shifting by +d and then by -d returns the keys to within the bf16
    rounding of two rotations, and the values exactly."""
    c = ShiftCase("bf16", "contiguous", 1, 1, 2, 128, 900, 0, seed=3)
    pb.pf_kv_shift(c.desc(100, 400, 300, 1e4), _stream())
    pb.pf_kv_shift(c.desc(400, 100, 300, 1e4), _stream())
    torch.cuda.synchronize()
    k1 = I.as_f64(_host(c.k, c.k0), "bf16")[0, 0, :, 100:400]
    k0 = I.as_f64(c.k0, "bf16")[0, 0, :, 100:400]
    v1 = _host(c.v, c.v0)[0, 0, :, 100:400]
    assert np.array_equal(v1, c.v0[0, 0, :, 100:400])
    assert np.max(np.abs(k1 - k0)) < 2.0 ** -6 * max(1.0, np.max(np.abs(k0)))


def test_kv_shift_full_size_window():
    """A 7B-VLM-shaped window move: 28 layers, 4 KV heads, D = 128, two
    retained 1300-token screenshots shifted down by one screenshot; sampled
    layers and heads checked."""
    c = ShiftCase("bf16", "contiguous", 28, 1, 4, 128, 4096, 0, seed=1)
    src, dst, count, base = 1400, 100, 2600, 1e6
    pb.pf_kv_shift(c.desc(src, dst, count, base), _stream())
    torch.cuda.synchronize()
    assert int(c.err.item()) == 0
    k1, v1 = _host(c.k, c.k0), _host(c.v, c.v0)
    for l in (0, 13, 27):
        K0 = I.as_f64(c.k0[l, 0], "bf16")
        Ko, _ = OR.shift_block(K0, K0, src, dst, count, base)
        got = I.as_f64(k1[l, 0], "bf16")[:, dst:dst + count]
        want = Ko[:, dst:dst + count]
        x = K0[:, src:src + count]
        pair = np.abs(x[..., :64]) + np.abs(x[..., 64:])
        tol = 2.0 ** -8 * np.abs(want) + 2.0 ** -20 * np.concatenate([pair, pair], -1)
        assert not (np.abs(got - want) > tol).any()
        assert np.array_equal(v1[l, 0, :, dst:dst + count], c.v0[l, 0, :, src:src + count])
        assert np.array_equal(k1[l, 0, :, dst + count:], c.k0[l, 0, :, dst + count:])


# ---------------------------------------------------------------------------
# pf_retrieval_key / pf_retrieve
# ---------------------------------------------------------------------------
def _workspace():
    n = pb.pf_retrieval_workspace_size()
    return torch.zeros(n, dtype=torch.uint8, device="cuda"), n


@pytest.mark.parametrize("dtype,H", [("bf16", 3584), ("bf16", 1536), ("f32", 4096),
                                     ("bf16", 100), ("f32", 1)])
def test_retrieval_key_matches_oracle(dtype, H):
    ws, n = _workspace()
    for rep in range(3):
        h = I.normal((H,), 1.0, rep, "key_hidden", H, dtype)
        P = I.normal((I.KEY_DIM, H), 1.0, 7, "key_projection", H, dtype)
        key = torch.zeros(I.KEY_DIM, dtype=torch.int8, device="cuda")
        hd, Pd = _dev(h), _dev(P)
        d = pb.pf_key_desc()
        d.dtype = pb.PF_BF16 if dtype == "bf16" else pb.PF_F32
        d.hidden, d.hidden_state, d.projection = H, hd.data_ptr(), Pd.data_ptr()
        d.key_out = key.data_ptr()
        pb.pf_retrieval_key(d, ws.data_ptr(), n, _stream())
        torch.cuda.synchronize()
        want, x = ORt.project_key(I.as_f64(h, dtype), I.as_f64(P, dtype))
        got = key.cpu().numpy()
        near = np.abs(np.abs(x - np.floor(x)) - 0.5) < 0.01
        assert np.array_equal(got[~near], want[~near])
        assert np.all(np.abs(got[near].astype(int) - want[near].astype(int)) <= 1)
        assert int(ws.count_nonzero().item()) == 0


def _retrieve(mem: I.Memory, qkey, token, lo=0, hi=None, dev=None):
    hi = len(mem.token) if hi is None else hi
    ws, n = _workspace()
    if dev is None:
        dev = dict(keys=_dev(mem.keys if len(mem.token) else np.zeros((1, 256), np.int8)),
                   token=_dev(mem.token if len(mem.token) else np.zeros(1, np.int32)),
                   pos=_dev(mem.pos if len(mem.token) else np.zeros(1, np.int32)),
                   bound=_dev(mem.bound if len(mem.token) else np.zeros(1, np.int32)))
    q = _dev(np.asarray(qkey, dtype=np.int8))
    best = torch.full((1,), -7, dtype=torch.int32, device="cuda")
    sim = torch.zeros(1, dtype=torch.float32, device="cuda")
    d = pb.pf_retrieval_desc()
    d.n_entries, d.lo, d.hi, d.token = len(mem.token), lo, hi, token
    d.query_key, d.keys = q.data_ptr(), dev["keys"].data_ptr()
    d.entry_token, d.entry_pos = dev["token"].data_ptr(), dev["pos"].data_ptr()
    d.entry_bound, d.best, d.similarity = dev["bound"].data_ptr(), best.data_ptr(), sim.data_ptr()
    pb.pf_retrieve(d, ws.data_ptr(), n, _stream())
    torch.cuda.synchronize()
    assert int(ws.count_nonzero().item()) == 0
    return int(best.item()), float(sim.item())


def _check_top1(mem, qkey, token, lo=0, hi=None):
    got_j, got_s = _retrieve(mem, qkey, token, lo, hi)
    want_j, want_s = ORt.cosine_top1(qkey, mem.keys, mem.token, mem.pos, mem.bound, token, lo, hi)
    assert got_j == want_j
    if want_j < 0:
        assert np.isnan(got_s)
    else:
        assert abs(got_s - want_s) <= 1e-6
    return got_j


@pytest.mark.parametrize("n", [1, 31, 33, 1000, 70001])
def test_retrieve_matches_oracle(n):
    mem = I.decoding_memory(n, seed=n)
    rng = np.random.default_rng(n)
    for rep in range(3):
        j = int(rng.integers(0, n))
        q = I.int8_keys(1, rep, "query_key", n)[0]
        _check_top1(mem, q, int(mem.token[j]))


def test_retrieve_paper_scale_memory():
    """~290K entries (the 74 MiB decoding memory of the paper's runs at 256 +
    12 bytes per entry); a frequent token, a rare token and a planted
    near-copy of an eligible entry's key."""
    n = 290000
    mem = I.decoding_memory(n, seed=11)
    tokens, counts = np.unique(mem.token, return_counts=True)
    frequent = int(tokens[np.argmax(counts)])
    rare = int(tokens[np.argmin(counts)])
    q = I.int8_keys(1, 0, "query_key", 1)[0]
    _check_top1(mem, q, frequent)
    _check_top1(mem, q, rare)
    elig = np.flatnonzero((mem.token == frequent) & (mem.pos < mem.bound))
    target = int(elig[len(elig) // 2])
    noisy = np.clip(mem.keys[target].astype(int) + I.int8_keys(1, 5, "noise")[0] // 20,
                    -127, 127).astype(np.int8)
    assert _check_top1(mem, noisy, frequent) == target


def test_retrieve_ties_ranges_and_empty():
    mem = I.decoding_memory(5000, seed=4)
    keys = mem.keys.copy()
    tok = mem.token.copy()
    pos, bound = mem.pos.copy(), mem.bound.copy()
    # an even query key, so that half of it is exact
    q = ((I.int8_keys(1, 9, "query_key")[0].astype(int) // 2) * 2).astype(np.int8)
    # exact duplicates of the query key at 4000 and 1500 (eligible): tie -> 1500;
    # the half-scaled copy at 700 has exactly the same cosine -> 700 wins
    for j in (4000, 1500):
        keys[j] = q
        tok[j] = 77
        bound[j] = pos[j] + 1
    keys[700] = (q.astype(int) // 2).astype(np.int8)
    tok[700] = 77
    bound[700] = pos[700] + 1
    # an all-zero eligible key is never selected; a boundary entry is skipped
    keys[10] = 0
    tok[10] = 77
    bound[10] = pos[10] + 1
    keys[20] = q
    tok[20] = 77
    bound[20] = pos[20]
    m2 = I.Memory(keys, tok, pos, bound)
    _check_top1(m2, q, 77)
    _check_top1(m2, q, 77, lo=701, hi=5000)   # only the duplicates: 1500
    _check_top1(m2, q, 77, lo=1501, hi=4001)  # 4000
    _check_top1(m2, q, 77, lo=21, hi=699)     # whatever else matches, or -1
    assert _check_top1(m2, q, 77, lo=10, hi=11) == -1
    assert _check_top1(m2, q, 77, lo=3, hi=3) == -1
    assert _check_top1(m2, q, -5) == -1
    empty = I.Memory(np.zeros((0, 256), np.int8), np.zeros(0, np.int32), np.zeros(0, np.int32),
                     np.zeros(0, np.int32))
    assert _check_top1(empty, q, 77) == -1


def test_retrieve_saturated_keys_need_wide_products():
    """Keys at +-127 make dot^2 * |k|^2 exceed 2^64 (about 7e19): the
    comparison must still be exact.  Entry 50 equals the query, entry 40 is
    the query with one sign flipped (slightly lower cosine), and entry 30 is
    the query with its first element set to 126 (higher cosine than 40,
    lower than 50)."""
    rng = np.random.default_rng(3)
    n = 100
    q = np.where(rng.random(256) < 0.5, -127, 127).astype(np.int8)
    keys = np.where(rng.random((n, 256)) < 0.5, -127, 127).astype(np.int8)
    keys[50] = q
    keys[40] = q
    keys[40, 7] = -q[7]
    keys[30] = q
    keys[30, 0] = 126 if q[0] > 0 else -126
    tok = np.full(n, 3, np.int32)
    pos = np.arange(n, dtype=np.int32)
    mem = I.Memory(keys, tok, pos, pos + 1)
    assert _check_top1(mem, q, 3) == 50
    assert _check_top1(mem, q, 3, lo=0, hi=50) == 30
    assert _check_top1(mem, q, 3, lo=31, hi=50) == 40


# ---------------------------------------------------------------------------
# pf_prefix_match
# ---------------------------------------------------------------------------
from oracle import prefix as OPX


def _prefix(prev, nxt, offset=0, with_len=True):
    """Run pf_prefix_match on device copies; `offset` elements of padding in
    front of each array make the pointers not 16-byte aligned."""
    pad = np.zeros(offset, dtype=np.int32)
    dp = torch.from_numpy(np.concatenate([pad, np.asarray(prev, np.int32)])).cuda()
    dn = torch.from_numpy(np.concatenate([pad, np.asarray(nxt, np.int32)])).cuda()
    out = torch.full((2,), -5, dtype=torch.int32, device="cuda")
    d = pb.pf_prefix_desc()
    d.prev = dp.data_ptr() + 4 * offset if len(prev) else None
    d.next = dn.data_ptr() + 4 * offset if len(nxt) else None
    d.n_prev, d.n_next = len(prev), len(nxt)
    d.lcp = out.data_ptr()
    d.cache_len = out.data_ptr() + 4 if with_len else None
    pb.pf_prefix_match(d, _stream())
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    if not with_len:
        assert got[1] == -5
    else:
        assert got[1] == got[0]
    return int(got[0])


@pytest.mark.parametrize("offset", [0, 1, 3])
def test_prefix_match_planted(offset):
    rng = np.random.default_rng(20 + offset)
    n = 40000
    a = rng.integers(0, 151936, size=n).astype(np.int32)
    for k in (0, 1, 3, 4, 4095, 4096, 4097, 8191, 12345, n - 1):
        b = a.copy()
        b[k] ^= 1 + int(rng.integers(0, 1000))
        b[k + 1:] = rng.integers(0, 151936, size=n - k - 1)
        want = OPX.common_prefix(a, b)
        assert want == k
        assert _prefix(a, b, offset) == want
        # other order, unequal lengths (the cut may remove the mismatch)
        assert _prefix(b[: n - 7], a, offset) == OPX.common_prefix(b[: n - 7], a)


def test_prefix_match_edges():
    rng = np.random.default_rng(7)
    a = rng.integers(-5, 5, size=9000).astype(np.int32)
    assert _prefix(a, a) == 9000                              # identical prompts
    assert _prefix(a, np.concatenate([a, a[:77]])) == 9000    # old prompt is a prefix
    assert _prefix(a[:4100], a) == 4100
    assert _prefix(a[:1], a[:1], offset=1) == 1
    assert _prefix([], a) == 0
    assert _prefix(a, []) == 0
    assert _prefix([], []) == 0
    assert _prefix(a, a, with_len=False) == 9000


def test_prefix_match_action_step_prompts():
    """Two consecutive action-step prompts of about 3.9K keys: shared system
    prompt and history, then a new screenshot (content keys) and question."""
    rng = np.random.default_rng(3)
    system = rng.integers(0, 151936, size=1200)
    hist = rng.integers(0, 151936, size=900)
    img_prev = (1 << 30) + rng.integers(0, 1 << 20, size=1300)   # content keys of a screenshot
    img_next = (1 << 30) + rng.integers(0, 1 << 20, size=1300)
    tail = rng.integers(0, 151936, size=500)
    prev = np.concatenate([system, hist, img_prev, tail]).astype(np.int32)
    nxt = np.concatenate([system, hist, img_next, tail]).astype(np.int32)
    want = OPX.common_prefix(prev, nxt)
    assert 2100 <= want < 2110
    assert _prefix(prev, nxt) == want
