"""Pins of the fp64 oracle to things other than itself.

Each ``pin_*`` function takes a loaded ``oracle.Oracle`` and raises
``AssertionError`` when the oracle disagrees with an independent statement of
the result:

* brute force over all K-subsets for the selection rule (Sec. 5.1 + Sec. 3.1);
* the counts of Fig. 1 and the sparsity 1 - s/G of Sec. 3.1;
* the worked example of Sec. 3.3 (``golden/sec3_3_example.txt``);
* Alg. 1 on the decompressed matrix against Alg. 2 taken literally, bit for bit
  on integer-valued inputs (Sec. 3.2);
* the K = G special case (no pruning), where the result must be the dense
  product, against ``torch.matmul`` in fp64;
* general K against ``torch.matmul`` / ``torch.nn.functional.conv2d`` in fp64 on
  the masked dense weights (library routines);
* 1x1 / stride 1 / pad 0 convolution equals the product;
* the error scale S against ``torch`` on |X| and |W|.

The same functions run against mutated builds of the oracle in
``test_oracle_mutants.py`` to show that each planted mistake is caught.  Run as
``python tests/oracle_pins.py LIB [LIB ...]`` to print, per library, the pins
that fail (used by the mutation test in a subprocess).
"""
from __future__ import annotations

import itertools
import json
import math
import os
import sys

import numpy as np
import torch
import torch.nn.functional as F

HERE = os.path.dirname(os.path.abspath(__file__))
if os.path.dirname(HERE) not in sys.path:
    sys.path.insert(0, os.path.dirname(HERE))

from oracle import Oracle, OracleError  # noqa: E402

GOLDEN = os.path.join(HERE, "golden")


def _rng(seed):
    return np.random.default_rng(seed)


def _read_fixture(name):
    out = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if not line or line.startswith("#"):
                continue
            key, *vals = line.split()
            out[key] = [float(v) for v in vals]
    return out


def _bruteforce_pack(W, G, K):
    """Exactly one K-subset has every kept j ahead of every dropped j' under the
    key (-|w|, j); return it for each (group, r)."""
    Cout, R = W.shape
    vals = np.zeros((Cout // G, R, K))
    idx = np.zeros((Cout // G, R, K), np.uint8)
    for gi in range(Cout // G):
        for r in range(R):
            col = [float(W[gi * G + j, r]) for j in range(G)]
            key = [(-abs(col[j]), j) for j in range(G)]
            found = []
            for sub in itertools.combinations(range(G), K):
                rest = [j for j in range(G) if j not in sub]
                if all(key[a] < key[b] for a in sub for b in rest):
                    found.append(sub)
            assert len(found) == 1, (gi, r, found)
            for s, j in enumerate(found[0]):
                vals[gi, r, s] = col[j]
                idx[gi, r, s] = j
    return vals, idx


def _same_bits(a, b):
    a = np.ascontiguousarray(a, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    return a.shape == b.shape and np.array_equal(a.view(np.int64), b.view(np.int64))


def pin_pack_bruteforce(orc: Oracle):
    rng = _rng(1)
    for G in (1, 2, 3, 4, 5, 6, 8):
        for K in range(1, G + 1):
            Cout, R = 2 * G, 6
            W = rng.integers(-3, 4, size=(Cout, R)).astype(np.float64)
            # signed zeros and infinities in a few places
            W[0, 0] = -0.0
            W[-1, 1] = np.inf
            W[min(1, Cout - 1), 2] = -np.inf
            W[:, 3] = -0.0 if G % 2 else 0.0
            v, i = orc.pack(W, G, K)
            ev, ei = _bruteforce_pack(W, G, K)
            assert np.array_equal(i, ei), (G, K)
            assert _same_bits(v, ev), (G, K)


def pin_fig1_counts(orc: Oracle):
    fx = _read_fixture("fig1_counts.txt")
    M, N, G, s = (int(fx[k][0]) for k in ("M", "N", "G", "s"))
    W = _rng(2).standard_normal((M, N))
    v, i = orc.pack(W, G, s)
    assert v.shape[0] * v.shape[2] == int(fx["compressed_rows"][0])
    assert v.shape[1] == N
    Wd, mask = orc.decompress(v, i, M, G)
    nz = int(np.count_nonzero(Wd))
    assert nz == int(fx["nonzeros"][0])
    assert Wd.size == int(fx["entries"][0])
    assert 1.0 - nz / Wd.size == fx["sparsity"][0]
    assert int(i.max()) < 2 ** int(fx["index_bits"][0])


def pin_sparsity_invariant(orc: Oracle):
    rng = _rng(3)
    for G, K in ((2, 1), (4, 1), (4, 3), (8, 2), (16, 4), (7, 3)):
        Cout, R = 4 * G, 11
        W = rng.standard_normal((Cout, R))
        v, i = orc.pack(W, G, K)
        Wd, mask = orc.decompress(v, i, Cout, G)
        per_group = np.count_nonzero(Wd.reshape(Cout // G, G, R), axis=1)
        assert np.all(per_group == K)
        assert math.isclose(1.0 - np.count_nonzero(Wd) / Wd.size, 1.0 - K / G)
        # kept magnitudes dominate dropped ones in every group
        A = np.abs(W).reshape(Cout // G, G, R)
        kept = mask.reshape(Cout // G, G, R) > 0
        assert np.all(np.where(kept, A, np.inf).min(axis=1) >= np.where(kept, -np.inf, A).max(axis=1))
        # kept values are the original weights, in increasing index
        assert np.all(np.diff(i.astype(int), axis=2) > 0)
        assert np.array_equal(Wd[mask > 0], W[mask > 0])


def pin_golden_sec33(orc: Oracle):
    fx = _read_fixture("sec3_3_example.txt")
    G, K = int(fx["G"][0]), int(fx["K"][0])
    W = np.array(fx["W_col0"]).reshape(G, 1)
    v, i = orc.pack(W, G, K)
    assert int(i[0, 0, 0]) == int(fx["expect_idx"][0])
    assert v[0, 0, 0] == fx["expect_value"][0]
    Wd, mask = orc.decompress(v, i, G, G)
    X = np.array(fx["X_row0"]).reshape(1, -1)  # N x columns, the paper's X
    Y, _ = orc.linear(X.T, Wd, mask)  # our layout: Y[column][channel] = H^T
    H = Y.T
    for row in range(G):
        assert np.array_equal(H[row], np.array(fx[f"expect_H_row{row}"])), row
    Y2 = orc.linear_alg2(X.T, v, i, G, G)
    assert np.array_equal(Y2.T, H)


def pin_alg1_eq_alg2_integer(orc: Oracle):
    rng = _rng(4)
    for G, K in ((1, 1), (4, 2), (8, 3), (6, 6), (16, 1)):
        Cout, R, N = 2 * G, 9, 7
        W = rng.integers(-4, 5, size=(Cout, R)).astype(np.float64)
        X = rng.integers(-4, 5, size=(N, R)).astype(np.float64)
        v, i = orc.pack(W, G, K)
        Wd, mask = orc.decompress(v, i, Cout, G)
        Y1, _ = orc.linear(X, Wd, mask)
        Y2 = orc.linear_alg2(X, v, i, Cout, G)
        assert np.array_equal(Y1, Y2), (G, K)
        # the same integers through a library matmul (exact in fp64 at these sizes)
        Yt = (torch.from_numpy(X) @ torch.from_numpy(Wd).T).numpy()
        assert np.array_equal(Y1, Yt), (G, K)


def pin_dense_special_case(orc: Oracle):
    rng = _rng(5)
    for G in (1, 4, 8):
        Cout, R, N = 3 * G, 13, 10
        W = rng.standard_normal((Cout, R))
        X = rng.standard_normal((N, R))
        v, i = orc.pack(W, G, G)  # K = G: nothing is pruned
        Wd, mask = orc.decompress(v, i, Cout, G)
        assert _same_bits(Wd, W) and np.all(mask == 1)
        Y, S = orc.linear(X, Wd, mask)
        Yt = (torch.from_numpy(X) @ torch.from_numpy(W).T).numpy()
        St = (torch.from_numpy(np.abs(X)) @ torch.from_numpy(np.abs(W)).T).numpy()
        assert np.all(np.abs(Y - Yt) <= 1e-12 * St)
        assert np.allclose(S, St, rtol=1e-12, atol=0)


def pin_linear_vs_torch(orc: Oracle):
    rng = _rng(6)
    for G, K, N, Cin, Cout in ((4, 2, 9, 17, 8), (8, 2, 5, 33, 16), (16, 4, 3, 40, 32),
                               (3, 1, 4, 7, 6)):
        W = rng.standard_normal((Cout, Cin))
        X = rng.uniform(-1, 1, size=(N, Cin))
        v, i = orc.pack(W, G, K)
        Wd, mask = orc.decompress(v, i, Cout, G)
        # masked dense weights built independently of the oracle: zero all but the
        # K largest |w| of each group column (ties cannot occur with continuous draws)
        A = np.abs(W).reshape(Cout // G, G, Cin)
        thresh = -np.sort(-A, axis=1)[:, K - 1:K, :]
        Wm = np.where(A >= thresh, W.reshape(Cout // G, G, Cin), 0.0).reshape(Cout, Cin)
        assert _same_bits(Wd, Wm)
        Y, S = orc.linear(X, Wd, mask)
        Yt = (torch.from_numpy(X) @ torch.from_numpy(Wm).T).numpy()
        St = (torch.from_numpy(np.abs(X)) @ torch.from_numpy(np.abs(Wm)).T).numpy()
        assert np.all(np.abs(Y - Yt) <= 1e-12 * St)
        assert np.allclose(S, St, rtol=1e-12, atol=0)


_CONV_CASES = (
    # B, H, W, Cin, Cout, KH, KW, stride, pad, G, K
    (2, 7, 6, 5, 8, 3, 3, (1, 1), (1, 1), 4, 2),
    (1, 9, 8, 3, 4, 3, 2, (2, 1), (1, 0), 2, 1),
    (2, 5, 5, 4, 8, 1, 1, (2, 2), (0, 0), 8, 3),
    (1, 6, 7, 2, 6, 5, 3, (1, 2), (2, 1), 3, 2),
    (1, 4, 4, 3, 4, 3, 3, (1, 1), (0, 0), 4, 4),
)


def pin_conv_vs_torch(orc: Oracle):
    rng = _rng(7)
    for (B, H, Wi, Cin, Cout, KH, KW, st, pd, G, K) in _CONV_CASES:
        W = rng.standard_normal((Cout, KH * KW * Cin))
        X = rng.standard_normal((B, H, Wi, Cin))
        v, i = orc.pack(W, G, K)
        Wd, mask = orc.decompress(v, i, Cout, G)
        Y, S = orc.conv2d(X, Wd, mask, KH, KW, st, pd)
        w4 = torch.from_numpy(Wd).reshape(Cout, KH, KW, Cin).permute(0, 3, 1, 2)
        x4 = torch.from_numpy(X).permute(0, 3, 1, 2)
        yt = F.conv2d(x4, w4, stride=st, padding=pd).permute(0, 2, 3, 1).reshape(-1, Cout).numpy()
        s4 = F.conv2d(x4.abs(), w4.abs(), stride=st, padding=pd)
        st_ = s4.permute(0, 2, 3, 1).reshape(-1, Cout).numpy()
        assert Y.shape == yt.shape
        assert np.all(np.abs(Y - yt) <= 1e-12 * st_ + 1e-300), (B, H, Wi, Cin, Cout, KH, KW)
        assert np.allclose(S, st_, rtol=1e-12, atol=0)
        # a subset of output positions gives the same rows
        pts = np.array([0, Y.shape[0] - 1, Y.shape[0] // 2], np.int64)
        Yp, _ = orc.conv2d(X, Wd, mask, KH, KW, st, pd, pts=pts)
        assert np.array_equal(Yp, Y[pts])


def pin_conv1x1_eq_linear(orc: Oracle):
    rng = _rng(8)
    B, H, Wi, Cin, Cout, G, K = 2, 3, 5, 6, 8, 4, 2
    W = rng.standard_normal((Cout, Cin))
    X = rng.standard_normal((B, H, Wi, Cin))
    v, i = orc.pack(W, G, K)
    Wd, mask = orc.decompress(v, i, Cout, G)
    Yc, Sc = orc.conv2d(X, Wd, mask, 1, 1)
    Yl, Sl = orc.linear(X.reshape(-1, Cin), Wd, mask)
    assert np.array_equal(Yc, Yl) and np.array_equal(Sc, Sl)


def pin_status_codes(orc: Oracle):
    W = np.ones((8, 3))
    W[3, 1] = np.nan
    try:
        orc.pack(W, 4, 2)
        raise AssertionError("NaN accepted")
    except OracleError as e:
        assert e.code == 6
    for G, K, Cout in ((0, 1, 8), (4, 5, 8), (3, 1, 8), (4, 0, 8), (257, 1, 257)):
        try:
            orc.pack(np.ones((Cout, 2)), G, K)
            raise AssertionError(f"bad group accepted {G} {K} {Cout}")
        except OracleError as e:
            assert e.code == 3


def pin_duplicate_idx(orc: Oracle):
    """A repeated index inside one (group, r) adds both values (what Alg. 2 does)."""
    G, K, Cout, R = 4, 2, 4, 3
    values = np.array([[[1.0, 2.0], [3.0, -1.0], [5.0, 7.0]]])
    idx = np.array([[[1, 1], [0, 3], [2, 2]]], np.uint8)
    Wd, mask = orc.decompress(values, idx, Cout, G)
    expect = np.zeros((Cout, R))
    expect[1, 0] = 3.0
    expect[0, 1], expect[3, 1] = 3.0, -1.0
    expect[2, 2] = 12.0
    assert np.array_equal(Wd, expect)
    assert mask[1, 0] == 2 and mask[2, 2] == 2
    X = np.array([[1.0, 2.0, 3.0], [-2.0, 0.5, 4.0]])
    Y1, _ = orc.linear(X, Wd, mask)
    Y2 = orc.linear_alg2(X, values, idx, Cout, G)
    assert np.array_equal(Y1, Y2)
    assert np.array_equal(Y1, X @ expect.T)


ALL_PINS = [
    pin_pack_bruteforce,
    pin_fig1_counts,
    pin_sparsity_invariant,
    pin_golden_sec33,
    pin_alg1_eq_alg2_integer,
    pin_dense_special_case,
    pin_linear_vs_torch,
    pin_conv_vs_torch,
    pin_conv1x1_eq_linear,
    pin_status_codes,
    pin_duplicate_idx,
]


def failing_pins(orc: Oracle):
    failed = []
    for pin in ALL_PINS:
        try:
            pin(orc)
        except Exception as e:  # noqa: BLE001 - any failure counts as caught
            failed.append(f"{pin.__name__}: {type(e).__name__}")
    return failed


if __name__ == "__main__":
    report = {lib: failing_pins(Oracle(lib)) for lib in sys.argv[1:]}
    print(json.dumps(report))
