"""Runtime-adaptive proposal-length controller (Section 3.2, eq. 1).

    L* = argmin_{0 <= l <= l_max}  T(l) / (A(l, s) + 1)

T(l): estimated latency of a decoding iteration that verifies l proposal
tokens; A(l, s): expected number of accepted proposal tokens at length l
and retrieval similarity s; the + 1 is the model token every iteration
appends.  l = 0 is an ordinary greedy pass.

Estimators (the paper names their form, not their details; readings):
  * acceptance: two online logistic regressions on x = (1, l / l_max, s),
    one for the probability p1 that the first proposal token is accepted,
    one for the probability pc that token k is accepted given token k - 1
    was; A(l, s) = sum_{k=1..l} p1 pc^(k-1).  One observation (l, s, a)
    gives one first-token trial (success iff a >= 1) and, when a >= 1, the
    continuation trials k = 2 .. min(a + 1, l) (success iff k <= a); each
    trial is one gradient step w += lr (y - sigmoid(w.x)) x.
  * latency: log T(l) = c0 + c1 u + c2 u^2 with u = l / l_max, fitted by
    recursive least squares from a zero prior of variance 1e8 per
    coefficient (least squares up to a relative bias of about 1e-8).
  * ties in the objective go to the shortest length; "occasionally explores
    an adjacent length": with the caller's uniform draw u < epsilon the
    choice moves to L* + 1 (or L* - 1 at l_max), the direction given by a
    second draw.

Test infrastructure only: imported by tests, never by the library.
"""
import math


def expected_accepted(p1, pc, ell):
    """A(l) = sum_{k=1..l} p1 * pc^(k-1), summed term by term."""
    return sum(p1 * pc ** (k - 1) for k in range(1, ell + 1))


def select_length(t_hat, p1, pc, l_max):
    """Eq. 1 over explicit per-length estimates: t_hat[l], p1[l], pc[l] for
    l = 0..l_max.  Returns (L*, objective at L*)."""
    best, best_obj = 0, None
    for ell in range(l_max + 1):
        obj = t_hat[ell] / (expected_accepted(p1[ell], pc[ell], ell) + 1.0)
        if best_obj is None or obj < best_obj:
            best, best_obj = ell, obj
    return best, best_obj


def _sigmoid(z):
    return 1.0 / (1.0 + math.exp(-z))


class AcceptanceModel:
    def __init__(self, l_max, lr):
        self.l_max, self.lr = l_max, lr
        self.w1 = [0.0, 0.0, 0.0]
        self.wc = [0.0, 0.0, 0.0]

    def _x(self, ell, s):
        return [1.0, ell / self.l_max, s]

    def predict(self, ell, s):
        x = self._x(ell, s)
        return (_sigmoid(sum(a * b for a, b in zip(self.w1, x))),
                _sigmoid(sum(a * b for a, b in zip(self.wc, x))))

    @staticmethod
    def _step(w, x, y, lr):
        g = y - _sigmoid(sum(a * b for a, b in zip(w, x)))
        for i in range(3):
            w[i] += lr * g * x[i]

    def update(self, ell, s, accepted):
        if ell < 1:
            return
        x = self._x(ell, s)
        self._step(self.w1, x, 1.0 if accepted >= 1 else 0.0, self.lr)
        if accepted >= 1:
            for k in range(2, min(accepted + 1, ell) + 1):
                self._step(self.wc, x, 1.0 if k <= accepted else 0.0, self.lr)


class LatencyModel:
    """Recursive least squares for log T = c . (1, l/l_scale, (l/l_scale)^2)
    (the scaled length keeps the normal equations well conditioned)."""

    def __init__(self, l_scale=128, prior_var=1e8):
        self.l_scale = l_scale
        self.c = [0.0, 0.0, 0.0]
        self.P = [[prior_var if i == j else 0.0 for j in range(3)] for i in range(3)]
        self.n = 0

    def _x(self, ell):
        u = ell / self.l_scale
        return [1.0, u, u * u]

    def update(self, ell, t):
        x = self._x(ell)
        y = math.log(t)
        Px = [sum(self.P[i][j] * x[j] for j in range(3)) for i in range(3)]
        denom = 1.0 + sum(x[i] * Px[i] for i in range(3))
        k = [v / denom for v in Px]
        err = y - sum(self.c[i] * x[i] for i in range(3))
        self.c = [self.c[i] + k[i] * err for i in range(3)]
        self.P = [[self.P[i][j] - k[i] * Px[j] for j in range(3)] for i in range(3)]
        self.n += 1

    def predict(self, ell):
        x = self._x(ell)
        return math.exp(self.c[0] * x[0] + self.c[1] * x[1] + self.c[2] * x[2])


def choose(lat, acc, s, l_max, u=1.0, u_dir=0.0, epsilon=0.0):
    """lat: a LatencyModel with l_scale = l_max."""
    """The controller's choice for similarity s from the two estimators."""
    t = [lat.predict(ell) for ell in range(l_max + 1)]
    pr = [acc.predict(ell, s) for ell in range(l_max + 1)]
    best, obj = select_length(t, [p[0] for p in pr], [p[1] for p in pr], l_max)
    if u < epsilon and l_max > 0:
        if best == 0 or (best < l_max and u_dir < 0.5):
            best += 1
        else:
            best -= 1
    return best, obj
