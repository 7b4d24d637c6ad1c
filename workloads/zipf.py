"""Zipf(alpha) sampler over ranks 1..N by rejection-inversion.

Method: Hormann & Derflinger, "Rejection-inversion to generate variates from
monotone discrete distributions", ACM TOMACS 6(3), 1996.  Restated here:
h(x) = x^-alpha is convex and decreasing on x > 0, so for every integer k the
area under h over [k - 1/2, k + 1/2] is at least the bar h(k).  Draw V uniform
on [H(1/2), H(N + 1/2)], where H is an antiderivative of h, and invert:
X = H^-1(V), k = round(X).  V lands in the slice [H(k + 1/2) - h(k),
H(k + 1/2)] of k's interval with probability proportional to h(k); accept
exactly then.  No O(N) table is needed, so N may be 4e8.

This is an input generator only: it holds none of the store's arithmetic.
"""
import math

import numpy as np


class ZipfSampler:
    """P(k) proportional to k^-alpha for k in 1..n (alpha > 0; alpha <= 1 allowed)."""

    def __init__(self, n: int, alpha: float):
        if n < 1 or alpha <= 0:
            raise ValueError("need n >= 1 and alpha > 0")
        self.n = int(n)
        self.a = float(alpha)
        self.lo = float(self._H(np.array([0.5]))[0])
        self.hi = float(self._H(np.array([self.n + 0.5]))[0])

    # H(x) = (x^(1-a) - 1) / (1-a), with the a -> 1 limit log(x).  Where
    # (1-a) log x is tiny the closed form loses digits and a series is used.
    def _H(self, x):
        lx = np.log(x)
        if self.a == 1.0:
            return lx
        t = (1.0 - self.a) * lx
        out = np.expm1(t) / (1.0 - self.a)
        small = np.abs(t) < 1e-8
        if np.any(small):
            ls, ts = lx[small], t[small]
            out[small] = ls * (1.0 + ts * (0.5 + ts / 6.0))
        return out

    def _Hinv(self, y):
        if self.a == 1.0:
            return np.exp(y)
        t = (1.0 - self.a) * y
        out = np.exp(np.log1p(t) / (1.0 - self.a))
        small = np.abs(t) < 1e-8
        if np.any(small):
            ys, ts = y[small], t[small]
            out[small] = np.exp(ys * (1.0 - ts * (0.5 - ts / 3.0)))
        return out

    def _h(self, k):
        return np.exp(-self.a * np.log(k))

    def sample(self, rng: np.random.Generator, size: int) -> np.ndarray:
        """`size` ranks in 1..n (int64), in draw order."""
        with np.errstate(over="ignore", divide="ignore", invalid="ignore"):
            return self._sample(rng, size)

    def _sample(self, rng, size):
        out = np.empty(size, np.int64)
        filled = 0
        while filled < size:
            m = int((size - filled) * 1.1) + 64
            v = self.lo + rng.random(m) * (self.hi - self.lo)
            x = self._Hinv(v)
            k = np.clip(np.floor(x + 0.5), 1, self.n)
            accept = v >= self._H(k + 0.5) - self._h(k)
            got = k[accept].astype(np.int64)
            take = min(len(got), size - filled)
            out[filled:filled + take] = got[:take]
            filled += take
        return out

    def pmf(self, ks) -> np.ndarray:
        """Exact probabilities (for tests on small n)."""
        ks = np.asarray(ks, np.float64)
        norm = math.fsum(float(r) ** -self.a for r in range(1, self.n + 1))
        return ks ** -self.a / norm


def scatter_bijection(n: int, rng: np.random.Generator):
    """A fixed bijection rank (1..n) -> index (0..n-1): (a (r-1) + b) mod n, gcd(a, n) = 1.

    It spreads the hot ranks over the key range, so hot rows are not adjacent.
    """
    while True:
        a = int(rng.integers(1, max(n, 2))) | 1
        if math.gcd(a, n) == 1:
            break
    b = int(rng.integers(0, n))

    def f(ranks: np.ndarray) -> np.ndarray:
        r = np.asarray(ranks, np.int64) - 1
        return (a * r + b) % n if n > 1 else np.zeros_like(r)

    return f
