"""The library's eq. 1 controller (host code, no GPU) against the oracle's:
same selections and the same estimator states on the same observations."""
import math

import numpy as np
import pytest

from oracle import controller as CT
from paper_2609_32166_gb300 import _build
from paper_2609_32166_gb300 import binding as pb


@pytest.fixture(scope="module", autouse=True)
def built():
    _build.build()


def test_length_select_matches_oracle():
    rng = np.random.default_rng(0)
    for trial in range(200):
        L = int(rng.integers(0, 70))
        t = 250 + np.cumsum(rng.random(L + 1) * 5)
        p1 = rng.random(L + 1)
        pc = rng.random(L + 1)
        got = pb.pf_length_select(t, p1, pc)
        want = CT.select_length(list(t), list(p1), list(pc), L)
        assert got[0] == want[0] and abs(got[1] - want[1]) <= 1e-12 * abs(want[1])


def test_length_select_pins():
    from tests import oracle_checks as C
    C.check_select_length_cases(lambda t, p1, pc, L: pb.pf_length_select(t, p1, pc))


def test_controller_tracks_the_oracle():
    rng = np.random.default_rng(1)
    L, lr, eps = 64, 0.05, 0.1
    c = pb.pf_controller_init(L, lr, eps)
    acc, lat = CT.AcceptanceModel(L, lr), CT.LatencyModel(L)
    for it in range(400):
        s = float(rng.random())
        u, ud = float(rng.random()), float(rng.random())
        got = pb.pf_controller_choose(c, s, u, ud)
        want = CT.choose(lat, acc, s, L, u, ud, eps)
        assert got[0] == want[0]
        assert abs(got[1] - want[1]) <= 1e-9 * abs(want[1])
        ell = got[0]
        a = int(rng.integers(0, ell + 1))
        t = math.exp(5.56 + 0.0043 * ell - 8.4e-6 * ell * ell) * (1 + 0.01 * rng.standard_normal())
        pb.pf_controller_observe(c, ell, s, a, t)
        acc.update(ell, s, a)
        lat.update(ell, t)
    assert np.allclose(list(c.w_first), acc.w1, rtol=1e-12, atol=1e-12)
    assert np.allclose(list(c.w_cont), acc.wc, rtol=1e-12, atol=1e-12)
    assert np.allclose(list(c.c), lat.c, rtol=1e-9, atol=1e-12)
    assert c.n_latency == lat.n == 400


def _train(c, accept_prob, latency, rng, n=3000):
    L = c.l_max
    for _ in range(n):
        s = float(rng.random())
        ell = int(rng.integers(1, L + 1))
        a = 0
        while a < ell and rng.random() < accept_prob(s):
            a += 1
        pb.pf_controller_observe(c, ell, s, a, latency(ell))


def test_controller_learns_to_propose_more_at_high_similarity():
    """Per-token acceptance that grows with similarity, latency rising 2 %
    per drafted token: the learned choice is longer for similar retrievals."""
    c = pb.pf_controller_init(32, 0.05, 0.0)
    _train(c, lambda s: 0.95 * s, lambda ell: 256.0 * (1 + 0.02 * ell), np.random.default_rng(2))
    hi = pb.pf_controller_choose(c, 0.95)[0]
    lo = pb.pf_controller_choose(c, 0.2)[0]
    assert hi > lo


def test_controller_falls_back_to_greedy_when_nothing_is_accepted():
    c = pb.pf_controller_init(32, 0.05, 0.0)
    _train(c, lambda s: 0.0, lambda ell: 256.0 * (1 + 0.01 * ell), np.random.default_rng(3))
    assert pb.pf_controller_choose(c, 0.99)[0] == 0


def test_controller_rejects_bad_arguments():
    with pytest.raises(pb.PfError):
        pb.pf_controller_init(0, 0.1, 0.0)
    with pytest.raises(pb.PfError):
        pb.pf_controller_init(8, 0.0, 0.0)
    c = pb.pf_controller_init(8, 0.1, 0.0)
    with pytest.raises(pb.PfError):
        pb.pf_controller_observe(c, 9, 0.5, 0, 1.0)
    with pytest.raises(pb.PfError):
        pb.pf_controller_observe(c, 4, 0.5, 5, 1.0)
