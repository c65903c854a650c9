"""Balanced sparsity, the paper's comparison format (Sec. 3.4): the oracle's
packing is pinned to a brute-force selection along the input dimension and its
decompression to the kept weights."""
import numpy as np
import pytest

import oracle


def brute(W, G, K):
    Cout, R = W.shape
    v = np.zeros((Cout, R // G, K))
    i = np.zeros((Cout, R // G, K), np.uint8)
    for co in range(Cout):
        for g in range(R // G):
            order = sorted(range(G), key=lambda j: (-abs(W[co, g * G + j]), j))[:K]
            for s, j in enumerate(sorted(order)):
                v[co, g, s] = W[co, g * G + j]
                i[co, g, s] = j
    return v, i


@pytest.mark.parametrize("Cout,R,G,K", [(5, 16, 4, 2), (3, 32, 8, 1), (7, 64, 16, 4), (2, 12, 3, 3)])
def test_bbs_pack_brute_force(Cout, R, G, K):
    rng = np.random.default_rng(Cout * R)
    W = np.round(rng.standard_normal((Cout, R)) * 3) / 3
    W[0, :2] = -0.0
    v, i = oracle.bbs_pack(W, G, K)
    vb, ib = brute(W, G, K)
    assert (i == ib).all()
    assert (v.view(np.int64) == vb.view(np.int64)).all()


def test_bbs_decompress_keeps_k_per_input_group():
    rng = np.random.default_rng(1)
    W = rng.standard_normal((6, 32))
    v, i = oracle.bbs_pack(W, 8, 2)
    Wd, mask = oracle.bbs_decompress(v, i, 32)
    assert (mask.reshape(6, 4, 8).sum(axis=2) == 2).all()           # exactly K per (co, input group)
    kept = mask.astype(bool)
    assert (Wd[kept] == W[kept]).all() and (Wd[~kept] == 0).all()
    # kept magnitudes dominate the dropped ones inside each group
    for co in range(6):
        for g in range(4):
            a = np.abs(W[co, g * 8:(g + 1) * 8])
            m = kept[co, g * 8:(g + 1) * 8]
            assert a[m].min() >= a[~m].max()


# ---------------------------------------------------------------------------
# the CUDA path: packing bit for bit, both product kernels within the tolerance
# ---------------------------------------------------------------------------
def _gpu():
    import torch
    from paper_1910_11971_gb300 import build as cci_build
    cci_build.build()
    return torch.device("cuda:0")


@pytest.mark.gpu
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("Cout,R,G,K", [(64, 256, 8, 2), (37, 96, 4, 1), (128, 1024, 16, 4), (8, 64, 32, 8),
                                        (3, 24, 3, 2)])
def test_bbs_pack_gpu(dtype, Cout, R, G, K):
    import torch
    import paper_1910_11971_gb300 as cci
    from parity_util import f64
    dev = _gpu()
    g = torch.Generator().manual_seed(Cout + R)
    W = (torch.randn((Cout, R), generator=g) * 2).round() / 2
    W[0, :3] = -0.0
    W = W.to(torch.float32 if dtype == "f32" else torch.bfloat16)
    v, i = cci.bbs_pack(W.to(dev), G, K)
    vo, io = oracle.bbs_pack(f64(W), G, K)
    assert (i.cpu().numpy() == io).all()
    assert (f64(v).view(np.int64) == vo.view(np.int64)).all()


@pytest.mark.gpu
@pytest.mark.parametrize("algo", ["tc", "gather"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,Cin,Cout,G,K", [(300, 256, 128, 8, 2), (129, 64, 68, 4, 1), (1000, 512, 256, 16, 4),
                                            (77, 96, 36, 32, 8)])
def test_bbs_linear_gpu(algo, dtype, N, Cin, Cout, G, K):
    import torch
    import paper_1910_11971_gb300 as cci
    from parity_util import assert_within_tol, f64
    dev = _gpu()
    g = torch.Generator().manual_seed(N + Cin)
    dt = torch.float32 if dtype == "f32" else torch.bfloat16
    X = torch.randn((N, Cin), generator=g).to(dt)
    W = torch.randn((Cout, Cin), generator=g).to(dt)
    v, i = cci.bbs_pack(W.to(dev), G, K)
    st = cci.new_status(dev)
    a = cci.ALGO_DENSE_TC_WS if algo == "tc" else cci.ALGO_GENERIC
    if algo == "tc" and dtype == "bf16" and Cin % 8:
        pytest.skip("tensor-core path needs Cin % 8")
    Y = cci.bbs_linear(X.to(dev), v, i, Cout, G, K, status=st, algo=a)
    assert cci.read_status(st) == 0
    vo, io = oracle.bbs_pack(f64(W), G, K)
    Wd, mask = oracle.bbs_decompress(vo, io, Cin)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, f"bbs {algo} {dtype} {N}x{Cin}->{Cout} G{G}K{K}")


@pytest.mark.gpu
def test_bbs_bad_index_reported():
    import torch
    import paper_1910_11971_gb300 as cci
    dev = _gpu()
    v = torch.ones((16, 8, 2), dtype=torch.bfloat16, device=dev)
    i = torch.zeros((16, 8, 2), dtype=torch.uint8, device=dev)
    i[..., 1] = 3
    i[2, 5, 1] = 9  # >= G
    X = torch.randn((40, 64), device=dev).to(torch.bfloat16)
    for algo in (cci.ALGO_DENSE_TC_WS, cci.ALGO_GENERIC):
        st = cci.new_status(dev)
        cci.bbs_linear(X, v, i, 16, 8, 2, status=st, algo=algo)
        assert cci.read_status(st) == 10
