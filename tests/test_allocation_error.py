"""Eq. 1 (Sec. 4): the probability P_d that a nonzero weight finds no encoding
slot.  The oracle's closed form is pinned to hand-worked values, to exact
enumeration of every zero pattern of a group, and to the trends the paper
states; its counting of dropped weights is pinned to its own packing."""
import itertools
from fractions import Fraction

import numpy as np
import pytest

import oracle


def test_hand_worked_values():
    # G = 2, Ps = 1/2, s = 1: only i = 2 overflows, B(2; 2, 1/2) = 1/4 -> P_d = 1/4
    assert oracle.allocation_error_exact(2, "1/2") == Fraction(1, 4)
    # G = 4, Ps = 1/2, s = 2: (1 * 4/16 + 2 * 1/16) / 2 = 3/16
    assert oracle.allocation_error_exact(4, "1/2") == Fraction(3, 16)
    assert oracle.allocation_error(4, 0.5) == pytest.approx(3 / 16, rel=1e-15)


def enumerate_pd(G: int, Ps: Fraction) -> Fraction:
    """Expected overflow over every zero pattern of one group, weighted by its
    probability, over the expected nonzeros: the definition behind Eq. 1."""
    p = 1 - Ps
    s = int(G * p)
    over = Fraction(0)
    for pattern in itertools.product((0, 1), repeat=G):
        nz = sum(pattern)
        over += max(nz - s, 0) * p ** nz * Ps ** (G - nz)
    return over / (G * p)


@pytest.mark.parametrize("G,Ps", [(2, "1/2"), (4, "1/2"), (4, "3/4"), (8, "3/4"), (8, "7/8"), (6, "2/3"),
                                  (10, "1/2"), (8, "1/4")])
def test_closed_form_equals_enumeration(G, Ps):
    exact = oracle.allocation_error_exact(G, Ps)
    assert exact == enumerate_pd(G, Fraction(Ps))
    assert oracle.allocation_error(G, float(Fraction(Ps))) == pytest.approx(float(exact), rel=1e-12)


def test_trends_stated_in_the_paper():
    """At a fixed sparsity P_d falls as G grows; at a fixed G it rises with the
    sparsity (Sec. 4, Fig. 3a)."""
    for Ps in ("1/2", "3/4", "7/8", "15/16"):
        q = Fraction(Ps).denominator
        gs = [g for g in (2, 4, 8, 16, 32, 64, 128, 256, 512, 1024) if g % q == 0]
        vals = [oracle.allocation_error_exact(g, Ps) for g in gs]
        assert all(a > b for a, b in zip(vals, vals[1:])), Ps
    for G in (16, 64, 256):
        vals = [oracle.allocation_error_exact(G, Ps) for Ps in ("1/2", "3/4", "7/8", "15/16")]
        assert all(a < b for a, b in zip(vals, vals[1:])), G


def sparse_weights(rng, Cout, R, Ps, dtype=np.float64):
    W = rng.standard_normal((Cout, R)).astype(dtype)
    W[rng.random((Cout, R)) < Ps] = 0
    return W


def test_pack_stats_equals_what_pack_drops():
    """Dropped nonzeros counted per group equal the nonzeros that the oracle's
    packing loses (nonzeros of W minus nonzeros of its decompression)."""
    rng = np.random.default_rng(0)
    for Cout, R, G, K, Ps in [(64, 33, 8, 2, 0.75), (48, 17, 16, 4, 0.5), (32, 9, 4, 1, 0.6)]:
        W = sparse_weights(rng, Cout, R, Ps)
        W[0, :5] = -0.0
        nz, dropped = oracle.pack_stats(W, G, K)
        v, i = oracle.pack(W, G, K)
        Wd, _ = oracle.decompress(v, i, Cout, G)
        assert nz == int((W != 0).sum())
        assert dropped == nz - int((Wd != 0).sum())


def test_pack_stats_matches_eq1_statistically():
    """On independent zeros the counted ratio estimates Eq. 1 (within 5 standard
    errors of the per-group mean)."""
    rng = np.random.default_rng(1)
    G, Ps = 8, 0.75
    K = int(G * (1 - Ps))
    W = sparse_weights(rng, 256, 2048, Ps)
    nz = (W.reshape(-1, G, 2048) != 0).sum(axis=1)
    over = np.maximum(nz - K, 0).ravel()
    est = over.mean() / K
    se = over.std(ddof=1) / np.sqrt(over.size) / K
    assert abs(est - oracle.allocation_error(G, Ps)) < 5 * se
    total_nz, dropped = oracle.pack_stats(W, G, K)
    assert dropped == int(over.sum())


def test_golden_table_is_the_oracle():
    """tests/golden/eq1_pd.txt (read by the benchmark) holds the oracle's values."""
    import os
    path = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden", "eq1_pd.txt")
    n = 0
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        Ps, G, s, pd = line.split()
        assert float(pd) == float(oracle.allocation_error_exact(int(G), Ps))
        assert int(s) == int(int(G) * (1 - Fraction(Ps)))
        n += 1
    assert n == 34  # 10 + 9 + 8 + 7 group sizes with an integer number of slots
