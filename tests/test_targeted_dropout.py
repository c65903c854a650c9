"""Targeted dropout for CCI training (Sec. 5.1): the oracle is pinned to a
brute-force statement on small inputs, to its end points (rate 0 keeps every
weight, rate 1 keeps exactly what packing keeps) and to the drop frequency; the
CUDA kernel matches it bit for bit on the GPU."""
import numpy as np
import pytest
import torch

import oracle
import paper_1910_11971_gb300 as cci
from parity_util import f64


def brute_force(W, G, K, rate, u):
    Cout, R = W.shape
    Wo, mask = W.copy(), np.ones((Cout, R), np.uint8)
    for gi in range(Cout // G):
        for r in range(R):
            order = sorted(range(G), key=lambda j: (-abs(W[gi * G + j, r]), j))
            for j in order[K:]:  # the candidates
                if np.float32(u[gi * G + j, r]) < np.float32(rate):
                    Wo[gi * G + j, r] = 0.0
                    mask[gi * G + j, r] = 0
    return Wo, mask


@pytest.mark.parametrize("G,K,rate", [(4, 2, 0.5), (8, 2, 0.73), (8, 1, 0.0), (16, 4, 1.0), (3, 1, 0.25)])
def test_oracle_equals_brute_force(G, K, rate):
    rng = np.random.default_rng(G * 10 + K)
    Cout, R = 4 * G, 11
    W = np.round(rng.standard_normal((Cout, R)) * 4) / 4  # many ties
    W[0, :3] = -0.0
    u = rng.random((Cout, R)).astype(np.float32)
    Wo, m = oracle.td_mask(W, G, K, rate, u)
    Wb, mb = brute_force(W, G, K, rate, u)
    assert (m == mb).all()
    assert (np.signbit(Wo) == np.signbit(Wb)).all() and (Wo == Wb).all()


def test_end_points():
    rng = np.random.default_rng(3)
    W = rng.standard_normal((32, 40))
    u = rng.random((32, 40)).astype(np.float32)
    Wo, m = oracle.td_mask(W, 8, 2, 0.0, u)
    assert (Wo == W).all() and m.all()
    Wo, m = oracle.td_mask(W, 8, 2, 1.0, u)
    v, i = oracle.pack(W, 8, 2)
    Wd, mask = oracle.decompress(v, i, 32, 8)
    assert (Wo == Wd).all() and (m == mask).all()


def test_drop_frequency():
    rng = np.random.default_rng(5)
    W = rng.standard_normal((256, 512))
    u = rng.random((256, 512)).astype(np.float32)
    _, m = oracle.td_mask(W, 8, 2, 0.6, u)
    cand = 256 * 512 * 6 // 8
    dropped = int((m == 0).sum())
    assert abs(dropped / cand - 0.6) < 5 * np.sqrt(0.6 * 0.4 / cand)


def test_drop_rate_schedule():
    """50 % at the start, 100 % at the end (Sec. 5.1), non-decreasing between (the
    library's host function; no device work)."""
    from paper_1910_11971_gb300 import build as cci_build
    cci_build.build()
    rates = [cci.td_drop_rate(s, 1000) for s in range(0, 1201, 50)]
    assert rates[0] == 0.5 and rates[-1] == 1.0 and cci.td_drop_rate(1000, 1000) == 1.0
    assert all(a <= b for a, b in zip(rates, rates[1:]))


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("Cout,R,G,K,rate", [(64, 37, 8, 2, 0.5), (96, 1000, 16, 4, 0.9), (4096, 1024, 8, 2, 0.75),
                                             (32, 9, 32, 8, 1.0), (12, 5, 4, 3, 0.0),
                                             (30, 41, 3, 1, 0.6), (128, 19, 64, 9, 0.8)])
def test_td_mask_matches_oracle(dtype, Cout, R, G, K, rate):
    from paper_1910_11971_gb300 import build as cci_build
    cci_build.build()
    dev = torch.device("cuda:0")
    g = torch.Generator().manual_seed(Cout + R)
    W = (torch.randn((Cout, R), generator=g) * 2).round() / 2  # ties
    W[0, :4] = -0.0
    W = W.to(dtype)
    u = torch.rand((Cout, R), generator=g)
    st = cci.new_status(dev)
    Wo, m = cci.td_mask(W.to(dev), G, K, rate, u.to(dev), status=st)
    assert cci.read_status(st) == 0
    Wr, mr = oracle.td_mask(f64(W), G, K, rate, u.numpy())
    assert (m.cpu().numpy() == mr).all()
    got = f64(Wo)
    assert (got == Wr).all() and (np.signbit(got) == np.signbit(Wr)).all()
