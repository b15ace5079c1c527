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


# ---------------------------------------------------------------------------
# eq. 1 driven by this library's own verify latency, measured on GB300
# ---------------------------------------------------------------------------
def _measured_curve():
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "verify_latency_curve.txt")
    pts = [tuple(float(x) for x in ln.split()) for ln in open(path)
           if ln.strip() and not ln.startswith("#")]
    return [(int(l), t) for l, t in pts]


def test_measured_curve_fits_identically():
    """Every measured (l, T) point fed to both controllers' latency models:
    the same log-quadratic coefficients, and a fit that follows the curve."""
    pts = _measured_curve()
    L = 127
    c = pb.pf_controller_init(L, 0.05, 0.0)
    lat = CT.LatencyModel(L)
    for ell, t in pts:
        pb.pf_controller_observe(c, ell, 0.0, -1, t)
        lat.update(ell, t)
    assert np.allclose(list(c.c), lat.c, rtol=1e-9, atol=1e-12)
    # the fitted model stays within 15 % of the measurement at every point
    for ell, t in pts:
        assert abs(lat.predict(ell) / t - 1.0) < 0.15, (ell, lat.predict(ell), t)


@pytest.mark.parametrize("q", [0.3, 0.6, 0.8, 0.9, 0.95, 0.99])
def test_measured_curve_same_choice_at_fixed_acceptance(q):
    """Eq. 1 on the fitted measured latency with a per-token acceptance q
    (p1 = pc = q): the library and the oracle pick the same length, and a
    higher acceptance never picks a shorter one."""
    pts = _measured_curve()
    L = 127
    c = pb.pf_controller_init(L, 0.05, 0.0)
    lat = CT.LatencyModel(L)
    for ell, t in pts:
        pb.pf_controller_observe(c, ell, 0.0, -1, t)
        lat.update(ell, t)
    u = np.arange(L + 1) / L
    t_lib = np.exp(c.c[0] + c.c[1] * u + c.c[2] * u * u)
    t_orc = [lat.predict(ell) for ell in range(L + 1)]
    got = pb.pf_length_select(t_lib, np.full(L + 1, q), np.full(L + 1, q))
    want = CT.select_length(t_orc, [q] * (L + 1), [q] * (L + 1), L)
    assert got[0] == want[0]
    assert abs(got[1] - want[1]) <= 1e-9 * want[1]
    lower = CT.select_length(t_orc, [q * 0.9] * (L + 1), [q * 0.9] * (L + 1), L)
    assert lower[0] <= want[0]


def test_measured_curve_online_controller_tracks_the_oracle():
    """The whole online controller on the measured latency: each iteration
    verifies at the chosen length, observes that length's measured T
    (linear between measured points) and a seeded Bernoulli acceptance
    outcome; the library and the oracle make the same choice every time."""
    pts = _measured_curve()
    xs, ys = np.array([p[0] for p in pts], float), np.array([p[1] for p in pts])
    L, lr, eps = 127, 0.05, 0.1
    rng = np.random.default_rng(5)
    c = pb.pf_controller_init(L, lr, eps)
    acc, lat = CT.AcceptanceModel(L, lr), CT.LatencyModel(L)
    for it in range(300):
        s = float(rng.random())
        uu, ud = float(rng.random()), float(rng.random())
        got = pb.pf_controller_choose(c, s, uu, ud)
        want = CT.choose(lat, acc, s, L, uu, ud, eps)
        assert got[0] == want[0], it
        ell = got[0]
        a = 0
        while a < ell and rng.random() < 0.5 + 0.45 * s:
            a += 1
        t = float(np.interp(ell, xs, ys))
        pb.pf_controller_observe(c, ell, s, a, t)
        acc.update(ell, s, a)
        lat.update(ell, t)
