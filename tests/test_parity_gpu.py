"""Parity of the CUDA path (through the C ABI) with the fp64 oracle.

* cci_pack: indices exact, values bit for bit, including ties, signed zeros and
  infinities (Sec. 5.1 selection, ties to the lower index).
* cci_linear / cci_conv2d: |y - y_oracle| <= 1e-5 * sum |w||x| per output, on
  small ragged shapes (all outputs) and at the full workload sizes in the
  launch configuration the benchmark times (sampled outputs: the first and
  last rows -- tile edges and the ragged tail -- and random ones).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_1910_11971_gb300 as cci
from paper_1910_11971_gb300 import build as cci_build
from paper_1910_11971_gb300 import workloads as wl
from parity_util import assert_pack_equal, assert_within_tol, f64, oracle_reference, sample_rows

pytestmark = pytest.mark.gpu

F32, BF16 = torch.float32, torch.bfloat16


@pytest.fixture(scope="module")
def dev():
    cci_build.build()
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    return torch.device("cuda:0")


def _dt(name):
    return F32 if name == "f32" else BF16


# ---------------------------------------------------------------------------
# pack
# ---------------------------------------------------------------------------
PACK_GK = [(1, 1), (2, 1), (3, 2), (4, 1), (4, 2), (4, 4), (5, 3), (8, 1), (8, 2), (8, 3), (8, 4),
           (16, 4), (16, 8), (32, 4), (32, 16), (64, 5), (256, 7), (256, 256)]


@pytest.mark.parametrize("R", [37, 40], ids=["R37", "R40_vec"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("G,K", PACK_GK)
def test_pack_random(dev, dtype, G, K, R):
    """R = 37: the one-column-per-thread kernels; R = 40: four columns per thread
    (vector loads) for the power-of-two G up to 32."""
    Cout = 2 * G
    W = wl.draw_w(Cout, R, 1.0, dtype, seed=G * 100 + K).to(dev)
    v, i = cci.pack(W, G, K)
    vo, io, _, _ = oracle_reference(W, G, K)
    assert_pack_equal(v, i, vo, io)


@pytest.mark.parametrize("R", [29, 32])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("G,K", [(4, 2), (8, 3), (16, 5), (3, 1), (32, 7)])
def test_pack_ties_signed_zero_inf(dev, dtype, G, K, R):
    Cout = 4 * G
    W = wl.integer_valued((Cout, R), -3, 3, seed=G + K)  # many equal magnitudes
    W[0, :5] = -0.0
    W[1, 5] = float("inf")
    W[2 % Cout, 6] = float("-inf")
    W[:, 7] = 0.0
    W[:, 8] = -0.0
    W = W.to(_dt(dtype)).to(dev)
    v, i = cci.pack(W, G, K)
    vo, io, _, _ = oracle_reference(W, G, K)
    assert_pack_equal(v, i, vo, io)


@pytest.mark.parametrize("R", [9, 12])
def test_pack_nan_reported(dev, R):
    W = torch.randn(16, R, device=dev)
    W[5, 3] = float("nan")
    with pytest.raises(cci.CCIError) as e:
        cci.pack(W, 8, 2)
    assert e.value.status == 6
    st = cci.new_status(dev)
    cci.pack(W.to(BF16), 8, 2, status=st, check=False)
    assert cci.read_status(st) == 6


@pytest.mark.parametrize("name", ["bottleneck_1x1", "conv3x3_28", "sweep_G32_K8", "resnet_l01"])
def test_pack_full_workloads(dev, name):
    if name == "bottleneck_1x1":
        case = wl.BOTTLENECK_1X1
        W = wl.draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed)
    elif name == "conv3x3_28":
        case = wl.CONV3X3_28
        W = wl.draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed)
    elif name == "sweep_G32_K8":
        case = wl.sweep_case(32, 8)
        W = wl.draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed)
    else:
        case = wl.resnet50_layers(K=2)[1]
        W = wl.draw_w(case.Cout, case.R, case.w_std, case.dtype, case.seed)
    v, i = cci.pack(W.to(dev), case.G, case.K)
    vo, io, _, _ = oracle_reference(W, case.G, case.K)
    assert_pack_equal(v, i, vo, io)


# ---------------------------------------------------------------------------
# products
# ---------------------------------------------------------------------------
def run_linear(dev, X, W, G, K, algo=cci.ALGO_AUTO):
    Xd, Wd_ = X.to(dev), W.to(dev)
    v, i = cci.pack(Wd_, G, K)
    Y = torch.full((X.shape[0], W.shape[0]), float("nan"), device=dev)  # poison: all must be written
    st = cci.new_status(dev)
    cci.linear(Xd, v, i, W.shape[0], G, K, out=Y, status=st, algo=algo)
    assert cci.read_status(st) == 0
    return Y


# (N, Cin, Cout, G, K, dtype): ragged N, N < tile, Cout = G, tiny Cin, and G / K
# without a register tile (generic kernel)
SMALL = [
    (1, 16, 8, 8, 2, "f32"), (33, 64, 64, 4, 2, "f32"), (257, 32, 16, 8, 1, "f32"),
    (300, 48, 24, 8, 4, "f32"), (1000, 16, 32, 16, 4, "f32"), (77, 64, 64, 32, 8, "f32"),
    (513, 256, 1024, 8, 2, "f32"), (130, 16, 64, 4, 1, "bf16"), (257, 64, 128, 16, 8, "bf16"),
    (96, 32, 64, 32, 16, "bf16"), (600, 128, 256, 8, 2, "bf16"), (45, 24, 16, 16, 2, "bf16"),
    (50, 20, 12, 3, 2, "f32"), (70, 12, 128, 64, 5, "bf16"), (9, 7, 256, 256, 3, "f32"),
    (65, 40, 16, 2, 1, "bf16"), (31, 64, 32, 8, 8, "f32"), (31, 64, 32, 8, 3, "bf16"),
]


@pytest.mark.parametrize("case", SMALL, ids=lambda c: "N{}_C{}x{}_G{}K{}_{}".format(*c))
def test_linear_small(dev, case):
    N, Cin, Cout, G, K, dtype = case
    X, W = wl.random_small(N + Cin, dtype, N, Cin, Cout)
    Y = run_linear(dev, X, W, G, K)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, str(case))


REGTILE_ALGOS = [cci.ALGO_REGTILE, cci.ALGO_EXPAND]


@pytest.mark.parametrize("algo", REGTILE_ALGOS, ids=["regtile", "expand"])
@pytest.mark.parametrize("case", [c for c in SMALL if c[0] > 1], ids=lambda c: "N{}_C{}x{}_G{}K{}_{}".format(*c))
def test_regtile_matches_generic_bitwise(dev, case, algo):
    """The kernels add the contributions of an output in the same order (ascending
    r, then slot, one FMA each, from +0); the expand kernel's extra terms are
    fma(0, x, acc) = acc exactly (acc is never -0), so all agree bit for bit."""
    N, Cin, Cout, G, K, dtype = case
    X, W = wl.random_small(N + 7 * Cin, dtype, N, Cin, Cout)
    name = cci.kernel_name(_dt(dtype), Cin, Cin, Cout, G, K, algo)
    if not name:
        pytest.skip("no register tile for this (G, K, dtype, shape)")
    Ya = run_linear(dev, X, W, G, K, algo)
    Yg = run_linear(dev, X, W, G, K, cci.ALGO_GENERIC)
    assert torch.equal(Ya.view(torch.int32), Yg.view(torch.int32))


def test_linear_tiny_workload(dev):
    case = wl.TINY_LINEAR
    X, W = wl.linear_inputs(case)
    Y = run_linear(dev, X, W, case.G, case.K)
    _, _, Wd, mask = oracle_reference(W, case.G, case.K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, case.name)


FULL_FAMILIES = [(cci.ALGO_AUTO, "dense_tc"), (cci.ALGO_REGTILE, "regtile"), (cci.ALGO_EXPAND, "expand")]


@pytest.mark.parametrize("algo,prefix", FULL_FAMILIES, ids=["auto", "regtile", "expand"])
def test_linear_bottleneck_full(dev, algo, prefix):
    """N = 100352 columns, 256 -> 1024, G=8, K=2, fp32: every output written;
    2048 sampled rows against the oracle.  AUTO through the binding (which
    passes a workspace) runs the tensor-core family; the two CUDA-core scatter
    families are selected explicitly."""
    case = wl.BOTTLENECK_1X1
    X, W = wl.linear_inputs(case)
    named = cci.ALGO_DENSE_TC_WS if algo == cci.ALGO_AUTO else algo
    assert cci.kernel_name(F32, case.Cin, case.R, case.Cout, case.G, case.K, named).startswith(prefix)
    Y = run_linear(dev, X, W, case.G, case.K, algo)
    assert torch.isfinite(Y).all()
    rows = sample_rows(case.N, 2048)
    _, _, Wd, mask = oracle_reference(W, case.G, case.K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, case.name)


@pytest.mark.parametrize("G,K", wl.SWEEP_POINTS)
def test_linear_sweep_full(dev, G, K):
    """4096 -> 4096, N = 8192, bf16: 192 sampled rows per (G, K) against the oracle."""
    case = wl.sweep_case(G, K)
    X, W = wl.linear_inputs(case, device="cpu")
    Y = run_linear(dev, X, W, G, K)
    assert torch.isfinite(Y).all()
    rows = sample_rows(case.N, 192, seed=G * 31 + K)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, case.name)


def test_linear_sweep_every_output_G8_K2(dev):
    """4096 -> 4096, N = 8192, bf16, G = 8, K = 2 through the production path:
    every one of the 33.5 M outputs against the oracle (about 69 GFLOP of fp64
    work on the host)."""
    case = wl.sweep_case(8, 2)
    X, W = wl.linear_inputs(case, device="cpu")
    Y = run_linear(dev, X, W, 8, 2)
    _, _, Wd, mask = oracle_reference(W, 8, 2)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, case.name + " (all outputs)")


@pytest.mark.parametrize("algo", [cci.ALGO_GENERIC] + REGTILE_ALGOS)
def test_linear_bad_index_reported(dev, algo):
    G, K, Cout, Cin, N = 8, 2, 16, 32, 40
    v = torch.ones((Cout // G, Cin, K), device=dev)
    i = torch.zeros((Cout // G, Cin, K), dtype=torch.uint8, device=dev)
    i[..., 1] = 1
    i[1, 5, 0] = 9  # >= G
    X = torch.randn(N, Cin, device=dev)
    st = cci.new_status(dev)
    cci.linear(X, v, i, Cout, G, K, status=st, algo=algo)
    assert cci.read_status(st) == 10


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("algo", [cci.ALGO_GENERIC] + REGTILE_ALGOS)
def test_linear_repeated_and_unordered_indices(dev, dtype, algo):
    """Packed input not produced by cci_pack: repeated and descending indices are
    summed as Alg. 2 does (the oracle's decompression sums them too)."""
    G, K, Cout, Cin, N = 8, 2, 32, 64, 300
    g = torch.Generator().manual_seed(3)
    v = torch.randn((Cout // G, Cin, K), generator=g).to(_dt(dtype))
    i = torch.randint(0, G, (Cout // G, Cin, K), generator=g, dtype=torch.uint8)
    X = torch.randn((N, Cin), generator=g).to(_dt(dtype))
    Y = cci.linear(X.to(dev), v.to(dev), i.to(dev), Cout, G, K, algo=algo)
    Wd, mask = oracle.decompress(f64(v), i.numpy(), Cout, G)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, "repeated indices")
    Y2 = oracle.linear_alg2(f64(X), f64(v), i.numpy(), Cout, G)
    assert_within_tol(f64(Y), Y2, S, "repeated indices vs Alg. 2")


def test_linear_empty(dev):
    v, i = cci.pack(torch.randn(16, 32, device=dev), 8, 2)
    Y = cci.linear(torch.empty((0, 32), device=dev), v, i, 16, 8, 2)
    assert Y.shape == (0, 16)


def test_linear_unaligned_views(dev):
    """Pointers off the 16-byte grid go to the generic kernel, with the same result."""
    G, K, Cout, Cin, N = 8, 2, 64, 32, 200
    X, W = wl.random_small(5, "f32", N + 1, Cin + 1, Cout)
    Xv = X.to(dev)[1:, 1:]  # not contiguous: make a contiguous copy shifted by one element
    base = torch.empty(N * Cin + 1, device=dev)
    base[1:].copy_(Xv.reshape(-1))
    Xs = base[1:].view(N, Cin)
    W = W[:, :Cin].contiguous()
    v, i = cci.pack(W.to(dev), G, K)
    Y = cci.linear(Xs, v, i, Cout, G, K)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(Xv), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, "unaligned")


# ---------------------------------------------------------------------------
# convolutions
# ---------------------------------------------------------------------------
def run_conv(dev, X, W, case_geom, G, K, algo=cci.ALGO_AUTO):
    KH, KW, stride, pad, Cout = case_geom
    v, i = cci.pack(W.to(dev), G, K)
    B, H, Wi, Cin = X.shape
    P, Q = cci.conv_out_hw(H, Wi, KH, KW, stride, pad)
    Y = torch.full((B, P, Q, Cout), float("nan"), device=dev)
    st = cci.new_status(dev)
    cci.conv2d(X.to(dev), v, i, Cout, G, K, KH, KW, stride, pad, out=Y, status=st, algo=algo)
    assert cci.read_status(st) == 0
    return Y


# (B, H, W, Cin, Cout, KH, KW, stride, pad, G, K, dtype)
CONV_SMALL = [
    (2, 9, 7, 16, 32, 3, 3, (1, 1), (1, 1), 8, 2, "bf16"),
    (1, 11, 10, 8, 16, 3, 3, (2, 2), (1, 1), 16, 4, "bf16"),
    (3, 6, 6, 32, 64, 1, 1, (2, 2), (0, 0), 8, 1, "bf16"),
    (2, 8, 5, 4, 16, 5, 3, (1, 2), (2, 1), 4, 2, "f32"),
    (1, 7, 7, 64, 128, 3, 3, (1, 1), (0, 0), 32, 8, "f32"),
    (2, 5, 5, 8, 8, 3, 3, (1, 1), (1, 1), 8, 4, "f32"),
    (1, 6, 9, 6, 12, 3, 2, (1, 1), (1, 0), 3, 2, "bf16"),  # generic kernel
    (4, 3, 3, 16, 64, 3, 3, (1, 1), (1, 1), 4, 1, "f32"),
]


@pytest.mark.parametrize("algo", [cci.ALGO_AUTO] + REGTILE_ALGOS, ids=["auto", "regtile", "expand"])
@pytest.mark.parametrize("case", CONV_SMALL, ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}_{}".format(*c))
def test_conv_small(dev, case, algo):
    B, H, Wi, Cin, Cout, KH, KW, stride, pad, G, K, dtype = case
    if not cci.kernel_name(_dt(dtype), Cin, KH * KW * Cin, Cout, G, K, algo):
        pytest.skip("no register tile for this (G, K, dtype, shape)")
    g = torch.Generator().manual_seed(B * 7 + Cin)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(_dt(dtype))
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(_dt(dtype))
    Y = run_conv(dev, X, W, (KH, KW, stride, pad, Cout), G, K, algo)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, stride, pad)
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, str(case))


def test_conv_1x1_equals_linear_bitwise(dev):
    B, H, Wi, Cin, Cout, G, K = 2, 14, 14, 64, 128, 8, 2
    X = torch.randn((B, H, Wi, Cin)).to(BF16)
    W = torch.randn((Cout, Cin)).to(BF16)
    Yc = run_conv(dev, X, W, (1, 1, (1, 1), (0, 0), Cout), G, K)
    Yl = run_linear(dev, X.reshape(-1, Cin), W, G, K)
    assert torch.equal(Yc.reshape(-1, Cout).view(torch.int32), Yl.view(torch.int32))


def conv_images(B: int, seed: int):
    """Images the sampled outputs come from: the first, the last, the middle one
    and a seeded interior one (4-D copy boxes span several images, so interior
    images sit inside boxes as well as on their edges)."""
    rng = np.random.default_rng(seed + 7)
    imgs = {0, B - 1, B // 2}
    if B > 3:
        imgs.add(int(rng.integers(1, B - 1)))
    return sorted(imgs)


def conv_points(case, k: int, seed: int, imgs):
    """Sampled output positions of the images `imgs` (as rows of the NHWC output):
    per image its first and last pixels (tile edges, the ragged tail) and random
    ones."""
    P, Q = case.P, case.Q
    per = P * Q
    rng = np.random.default_rng(seed)
    each = max(8, k // len(imgs))
    pts = []
    for b in imgs:
        edge = min(per, each // 4)
        pts.append(b * per + np.concatenate([np.arange(edge), np.arange(per - edge, per),
                                             rng.choice(per, size=each // 2)]))
    return np.unique(np.concatenate(pts))


def check_conv_case(dev, case, npts=1024, seed=0, algo=cci.ALGO_AUTO):
    X, W = wl.conv_inputs(case, device="cpu")
    Y = run_conv(dev, X, W, (case.KH, case.KW, (case.stride,) * 2, (case.pad,) * 2, case.Cout),
                 case.G, case.K, algo)
    assert torch.isfinite(Y).all()
    imgs = conv_images(case.B, seed)
    pts = conv_points(case, npts, seed, imgs)
    # oracle on the images the points come from, the points renumbered within them
    Xs = f64(X[imgs])
    per = case.P * case.Q
    pos = {b: j for j, b in enumerate(imgs)}
    local = np.array([pos[int(p) // per] * per + int(p) % per for p in pts], dtype=np.int64)
    _, _, Wd, mask = oracle_reference(W, case.G, case.K)
    Yo, S = oracle.conv2d(Xs, Wd, mask, case.KH, case.KW, (case.stride,) * 2, (case.pad,) * 2, pts=local)
    Yg = f64(Y.reshape(-1, case.Cout)[torch.from_numpy(pts).to(dev)])
    assert_within_tol(Yg, Yo, S, case.name)


@pytest.mark.parametrize("algo,prefix", FULL_FAMILIES, ids=["auto", "regtile", "expand"])
def test_conv3x3_full(dev, algo, prefix):
    """Batch 64, 28x28, 128 -> 128, 3x3 s1 p1, G=16, K=4, bf16, through AUTO (the
    tensor-core family) and the two CUDA-core scatter families explicitly."""
    case = wl.CONV3X3_28
    named = cci.ALGO_DENSE_TC_WS if algo == cci.ALGO_AUTO else algo
    name = cci.kernel_name(BF16, case.Cin, case.R, case.Cout, case.G, case.K, named)
    if not name:
        pytest.skip("no register tile for (G, K) = (16, 4) in bf16")
    assert name.startswith(prefix)
    check_conv_case(dev, case, npts=2048, algo=algo)


RESNET_PICK = [0, 1, 3, 4, 11, 13, 15, 24, 25, 28, 42, 44, 47, 49, 51]


@pytest.mark.parametrize("K", [1, 2, 4])
@pytest.mark.parametrize("li", RESNET_PICK)
def test_resnet50_layer(dev, li, K):
    """Layers of the ResNet-50 stack (batch 128), G=8: first/last 1x1, 3x3 s1 at
    every stage (56, 28, 14, 7) and s2, strided downsample 1x1."""
    case = wl.resnet50_layers(K=K)[li]
    check_conv_case(dev, case, npts=512, seed=li)


# ---------------------------------------------------------------------------
# dense tensor-core comparison kernel (tcgen05, bf16)
# ---------------------------------------------------------------------------
# (N, Cin, Cout, G, K): one tile, ragged N and Cout, several tiles per CTA, every (G, K) family
DENSE_SMALL = [
    (128, 64, 256, 8, 2), (1, 64, 256, 8, 2), (200, 64, 256, 8, 2), (300, 128, 512, 8, 2),
    (130, 72, 40, 4, 1), (257, 136, 96, 4, 2), (64, 64, 64, 16, 4), (515, 192, 384, 16, 8),
    (129, 80, 64, 32, 16), (100, 256, 320, 32, 4), (1000, 64, 256, 8, 4), (77, 8, 32, 16, 1),
    # reductions shorter than one 64-deep stage: the copies and MMAs cover R rounded up to 16
    (300, 16, 96, 8, 2), (1000, 24, 144, 8, 2), (257, 32, 16, 8, 2), (129, 40, 64, 8, 1), (64, 48, 128, 16, 4),
    (40000, 16, 96, 8, 2),
]


DENSE_ALGOS = [cci.ALGO_DENSE_TC, cci.ALGO_DENSE_TC_WS]
DENSE_IDS = ["fused", "ws"]


def skip_without(dtype, Cin, R, Cout, G, K, algo):
    name = cci.kernel_name(dtype, Cin, R, Cout, G, K, algo)
    if not name:
        pytest.skip("the family does not have this layer")
    assert name.startswith("dense_tc")


@pytest.mark.parametrize("algo", DENSE_ALGOS, ids=DENSE_IDS)
@pytest.mark.parametrize("case", DENSE_SMALL, ids=lambda c: "N{}_C{}x{}_G{}K{}".format(*c))
def test_dense_tc_small(dev, case, algo):
    N, Cin, Cout, G, K = case
    X, W = wl.random_small(N * 3 + Cin, "bf16", N, Cin, Cout)
    skip_without(BF16, Cin, Cin, Cout, G, K, algo)
    Y = run_linear(dev, X, W, G, K, algo)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, str(case))


@pytest.mark.parametrize("algo", DENSE_ALGOS, ids=DENSE_IDS)
@pytest.mark.parametrize("G,K", wl.SWEEP_POINTS)
def test_dense_tc_sweep_full(dev, G, K, algo):
    case = wl.sweep_case(G, K)
    skip_without(BF16, case.Cin, case.R, case.Cout, G, K, algo)
    X, W = wl.linear_inputs(case, device="cpu")
    Y = run_linear(dev, X, W, G, K, algo)
    assert torch.isfinite(Y).all()
    rows = sample_rows(case.N, 192, seed=G * 37 + K)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, case.name + " dense_tc")


@pytest.mark.parametrize("case", [c for c in CONV_SMALL if c[-1] == "bf16" and c[3] % 8 == 0 and c[9] in (4, 8, 16, 32)
                                  and (c[10] & (c[10] - 1)) == 0 and c[10] <= c[9] // 2],
                         ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}_{}".format(*c))
@pytest.mark.parametrize("algo", DENSE_ALGOS, ids=DENSE_IDS)
def test_dense_tc_conv_small(dev, case, algo):
    B, H, Wi, Cin, Cout, KH, KW, stride, pad, G, K, dtype = case
    if algo == cci.ALGO_DENSE_TC and not (Cin % 64 == 0 or (KH == KW == 1 and stride == (1, 1) and pad == (0, 0))):
        pytest.skip("fused family: activations by TMA need Cin % 64 == 0")
    g = torch.Generator().manual_seed(B * 11 + Cin)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (KH, KW, stride, pad, Cout), G, K, algo)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, stride, pad)
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, str(case))


@pytest.mark.parametrize("algo", DENSE_ALGOS, ids=DENSE_IDS)
def test_dense_tc_conv3x3_full(dev, algo):
    check_conv_case(dev, wl.CONV3X3_28, npts=1024, seed=5, algo=algo)


@pytest.mark.parametrize("algo", DENSE_ALGOS, ids=DENSE_IDS)
def test_dense_tc_rejects_repeated_indices(dev, algo):
    """A dense tile holds one weight per (channel, r): index sets must be strictly
    increasing (cci_pack's output); anything else is reported."""
    G, K, Cout, Cin, N = 8, 2, 256, 64, 128
    v = torch.ones((Cout // G, Cin, K), dtype=BF16, device=dev)
    i = torch.zeros((Cout // G, Cin, K), dtype=torch.uint8, device=dev)
    i[..., 1] = 3
    i[2, 7, 1] = 0  # repeated index
    X = torch.randn(N, Cin, device=dev).to(BF16)
    st = cci.new_status(dev)
    cci.linear(X, v, i, Cout, G, K, status=st, algo=algo)
    assert cci.read_status(st) == 10


# ---------------------------------------------------------------------------
# the fused tensor-core family: packed weights expanded inside the GEMM
# ---------------------------------------------------------------------------
# (N, Cin, Cout, G, K): ragged N, Cout below a tile (64-wide N tiles, idle
# producers), two-group items (G = 4), row blocks of larger groups (G = 16, 32),
# K = 8, a reduction not a multiple of the 64-deep stage (R = 80, 200, 136),
# long reductions (R up to 2048), groups past Cout in the last channel tile
# (Cout = 320, 96); the CTA-pair tiles are covered by the sweep tests
FUSED_SMALL = [
    (1, 64, 64, 8, 2), (129, 80, 96, 8, 1), (300, 200, 320, 4, 2), (257, 128, 128, 4, 1),
    (515, 192, 384, 16, 8), (100, 256, 320, 32, 4), (77, 64, 64, 32, 8), (640, 1024, 512, 8, 2),
    (1000, 2048, 1024, 16, 4), (333, 1088, 768, 32, 1), (4096, 512, 2048, 8, 4), (130, 136, 96, 16, 2),
]


@pytest.mark.parametrize("case", FUSED_SMALL, ids=lambda c: "N{}_C{}x{}_G{}K{}".format(*c))
def test_fused_small(dev, case):
    N, Cin, Cout, G, K = case
    skip_without(BF16, Cin, Cin, Cout, G, K, cci.ALGO_DENSE_TC)
    X, W = wl.random_small(N * 7 + Cin + G, "bf16", N, Cin, Cout)
    Y = run_linear(dev, X, W, G, K, cci.ALGO_DENSE_TC)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, "fused " + str(case))
    Yw = run_linear(dev, X, W, G, K, cci.ALGO_DENSE_TC_WS)
    assert_within_tol(f64(Y), f64(Yw), S, "fused vs workspace " + str(case))


# (B, H, W, Cin, Cout, KH, KW, stride, pad, G, K): 4-D copies at stride 1 and 2,
# a 1x1 stride-2 downsample, halo copies (3x3, Cin >= 256) with K = 8, a 5x5
# window, CTA pairs on a long reduction
FUSED_CONV = [
    (2, 14, 14, 64, 128, 3, 3, 1, 1, 8, 2), (3, 15, 15, 64, 64, 3, 3, 2, 1, 16, 4),
    (2, 14, 14, 128, 256, 1, 1, 2, 0, 8, 1), (1, 14, 14, 256, 256, 3, 3, 1, 1, 8, 4),
    (2, 7, 7, 512, 512, 3, 3, 1, 1, 32, 8), (2, 12, 12, 64, 64, 5, 5, 1, 2, 4, 2),
    (16, 14, 14, 256, 512, 3, 3, 2, 1, 8, 2), (8, 28, 28, 128, 128, 3, 3, 1, 1, 16, 4),
]


@pytest.mark.parametrize("case", FUSED_CONV, ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}".format(*c))
def test_fused_conv(dev, case):
    B, H, Wi, Cin, Cout, KH, KW, s_, p_, G, K = case
    skip_without(BF16, Cin, KH * KW * Cin, Cout, G, K, cci.ALGO_DENSE_TC)
    g = torch.Generator().manual_seed(B * 13 + Cin + KH)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (KH, KW, (s_, s_), (p_, p_), Cout), G, K, cci.ALGO_DENSE_TC)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, (s_, s_), (p_, p_))
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, "fused conv " + str(case))


def test_fused_checks_index_sets_of_every_tile(dev):
    """Many column tiles: the CTAs of the first column tile check every group's
    index sets, so a bad set anywhere is reported (an index >= G here, in the
    last group and the last reduction index)."""
    G, K, Cout, Cin, N = 8, 2, 512, 128, 2000
    W = torch.randn((Cout, Cin), device=dev).to(BF16)
    v, i = cci.pack(W, G, K)
    X = torch.randn(N, Cin, device=dev).to(BF16)
    st = cci.new_status(dev)
    cci.linear(X, v, i, Cout, G, K, status=st, algo=cci.ALGO_DENSE_TC)
    assert cci.read_status(st) == 0
    i[-1, -1, 1] = G
    st = cci.new_status(dev)
    cci.linear(X, v, i, Cout, G, K, status=st, algo=cci.ALGO_DENSE_TC)
    assert cci.read_status(st) == 10


def test_auto_without_workspace_uses_fused(dev):
    """Plain cci_linear (AUTO, no workspace) reaches the tensor cores through the
    fused family, with the workspace family's result."""
    N, Cin, Cout, G, K = 700, 256, 512, 8, 2
    X, W = wl.random_small(41, "bf16", N, Cin, Cout)
    Xd = X.to(dev)
    v, i = cci.pack(W.to(dev), G, K)
    assert cci.kernel_name(BF16, Cin, Cin, Cout, G, K, cci.ALGO_DENSE_TC).startswith("dense_tc_fused")
    Y = torch.empty((N, Cout), device=dev)
    st = cci.new_status(dev)
    code = cci.lib().cci_linear(Xd.data_ptr(), cci.BF16, N, Cin, v.data_ptr(), i.data_ptr(), Cout, G, K,
                                Y.data_ptr(), st.data_ptr(), torch.cuda.current_stream(dev).cuda_stream)
    assert code == 0 and cci.read_status(st) == 0
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, "plain cci_linear")


def test_auto_with_workspace_uses_dense_tc_ws(dev):
    """AUTO picks the workspace tensor-core family for a bf16 layer the fused
    family does not take (K = 8) when given a workspace."""
    N, Cin, Cout, G, K = 300, 64, 256, 16, 8
    X, W = wl.random_small(4, "bf16", N, Cin, Cout)
    Xd = X.to(dev)
    v, i = cci.pack(W.to(dev), G, K)
    ws = cci.new_workspace(cci.ALGO_AUTO, BF16, Cout, Cin, dev)
    assert ws is not None and ws.numel() == Cout * Cin * 2
    Ya = cci.linear(Xd, v, i, Cout, G, K, workspace=ws)
    Yw = cci.linear(Xd, v, i, Cout, G, K, algo=cci.ALGO_DENSE_TC_WS)
    assert torch.equal(Ya.view(torch.int32), Yw.view(torch.int32))


# ---------------------------------------------------------------------------
# fp32 on the tensor cores: the split product (tf32 hi*hi plus bf16 cross terms) through the workspace family
# ---------------------------------------------------------------------------
F32_DENSE = [(128, 64, 128, 8, 2), (1, 16, 128, 8, 2), (200, 36, 200, 4, 1), (300, 132, 384, 16, 4),
             (515, 64, 96, 32, 8), (129, 256, 1024, 8, 2), (77, 12, 64, 16, 8)]


@pytest.mark.parametrize("case", F32_DENSE, ids=lambda c: "N{}_C{}x{}_G{}K{}".format(*c))
def test_f32split_small(dev, case):
    N, Cin, Cout, G, K = case
    X, W = wl.random_small(N * 5 + Cin, "f32", N, Cin, Cout)
    assert cci.kernel_name(F32, Cin, Cin, Cout, G, K, cci.ALGO_DENSE_TC_WS).startswith("dense_tc_ws_f32split")
    Y = run_linear(dev, X, W, G, K, cci.ALGO_DENSE_TC_WS)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, str(case))


@pytest.mark.parametrize("algo", [cci.ALGO_DENSE_TC_WS, cci.ALGO_GENERIC], ids=["f32split", "generic"])
def test_fp32_wide_exponent_range(dev, algo):
    """Every activation row and every group of G output channels of W carries its
    own power-of-two scale (2^-30 .. 2^30), so the per-output scale S spans ~35 orders of
    magnitude: the product must hold |err| <= 1e-5 * S for each output (no absolute
    error floor; for the split product, hi, lo and their bf16 forms keep fp32's exponent
    range)."""
    N, Cin, Cout, G, K = 700, 256, 256, 8, 2
    g = torch.Generator().manual_seed(2024)
    X = torch.randn((N, Cin), generator=g) * torch.pow(2.0, torch.randint(-30, 31, (N, 1), generator=g).float())
    # one scale per group of G output channels: every channel keeps weights (a scale
    # per channel would let the two largest-scaled channels of a group win every r)
    wsc = torch.pow(2.0, torch.randint(-30, 31, (Cout // G, 1, 1), generator=g).float())
    W = (torch.randn((Cout // G, G, Cin), generator=g) * wsc).reshape(Cout, Cin)
    X[::7, ::5] = 0.0  # exact zeros among the activations (ReLU-like)
    Y = run_linear(dev, X, W, G, K, algo)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert float(S[S > 0].max() / S[S > 0].min()) > 1e30  # this draw: ~4e35
    assert_within_tol(f64(Y), Yo, S, "fp32 wide exponent range")


def test_f32split_bottleneck_full(dev):
    case = wl.BOTTLENECK_1X1
    X, W = wl.linear_inputs(case)
    Y = run_linear(dev, X, W, case.G, case.K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    rows = sample_rows(case.N, 2048, seed=3)
    _, _, Wd, mask = oracle_reference(W, case.G, case.K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, case.name + " f32split")


@pytest.mark.parametrize("case", [c for c in CONV_SMALL if c[-1] == "f32" and c[3] % 4 == 0 and c[9] in (4, 8, 16, 32)
                                  and (c[10] & (c[10] - 1)) == 0 and c[10] <= c[9] // 2],
                         ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}_{}".format(*c))
def test_f32split_conv_small(dev, case):
    B, H, Wi, Cin, Cout, KH, KW, stride, pad, G, K, dtype = case
    g = torch.Generator().manual_seed(B * 13 + Cin)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0)
    W = torch.randn((Cout, KH * KW * Cin), generator=g)
    Y = run_conv(dev, X, W, (KH, KW, stride, pad, Cout), G, K, cci.ALGO_DENSE_TC_WS)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, stride, pad)
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, str(case))


# ---------------------------------------------------------------------------
# convolutions whose activations are copied by 4-D TMA (strides 1 or 2, Cin a
# multiple of 64 for bf16 / 32 for fp32): output-pixel boxes with ragged edges,
# asymmetric padding, windows wholly inside the padding, every N tile width
# ---------------------------------------------------------------------------
# (B, H, W, Cin, Cout, KH, KW, stride, pad, G, K, dtype)
CONV_TMA = [
    (3, 9, 7, 64, 64, 3, 3, (1, 1), (1, 1), 8, 2, "bf16"),
    (2, 13, 11, 128, 192, 3, 3, (1, 1), (1, 1), 16, 4, "bf16"),
    (1, 6, 20, 64, 32, 5, 3, (1, 1), (2, 0), 4, 2, "bf16"),
    (5, 7, 7, 64, 128, 3, 3, (1, 1), (0, 0), 8, 4, "bf16"),
    (2, 4, 4, 64, 64, 3, 3, (1, 1), (3, 3), 8, 1, "bf16"),
    (2, 5, 5, 64, 64, 1, 1, (1, 1), (1, 1), 8, 2, "bf16"),
    (33, 3, 5, 192, 256, 3, 3, (1, 1), (1, 1), 32, 8, "bf16"),
    (2, 9, 7, 32, 64, 3, 3, (1, 1), (1, 1), 8, 2, "f32"),
    (3, 5, 6, 64, 96, 3, 3, (1, 1), (1, 1), 16, 4, "f32"),
    (2, 4, 4, 32, 32, 3, 3, (1, 1), (3, 3), 4, 1, "f32"),
    # strides 2: one copy map per parity lattice of the input
    (2, 9, 7, 64, 64, 3, 3, (2, 2), (1, 1), 8, 2, "bf16"),
    (3, 8, 10, 64, 128, 1, 1, (2, 2), (0, 0), 8, 2, "bf16"),
    (2, 7, 6, 128, 64, 3, 3, (2, 1), (1, 0), 16, 4, "bf16"),
    (1, 5, 5, 64, 32, 5, 5, (2, 2), (2, 2), 4, 1, "bf16"),
    (2, 2, 3, 64, 64, 3, 3, (2, 2), (1, 1), 8, 2, "bf16"),
    (2, 9, 7, 32, 64, 3, 3, (2, 2), (1, 1), 8, 2, "f32"),
    (2, 6, 6, 32, 32, 1, 1, (2, 2), (0, 0), 4, 2, "f32"),
    # stride 3: the row gather
    (1, 10, 10, 64, 64, 3, 3, (3, 3), (1, 1), 8, 2, "bf16"),
]


@pytest.mark.parametrize("case", CONV_TMA, ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}_{}".format(*c))
def test_dense_tc_ws_conv_tma(dev, case):
    B, H, Wi, Cin, Cout, KH, KW, stride, pad, G, K, dtype = case
    g = torch.Generator().manual_seed(B * 17 + Cin + Cout)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(_dt(dtype))
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(_dt(dtype))
    Y = run_conv(dev, X, W, (KH, KW, stride, pad, Cout), G, K, cci.ALGO_DENSE_TC_WS)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, stride, pad)
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, str(case))


def test_dense_tc_ws_conv_tma_equals_gather_bitwise(dev):
    """A convolution whose activations arrive by 4-D copy equals, bit for bit,
    the product of its im2col matrix (2-D copy): same operands, same order."""
    B, H, Wi, Cin, Cout, G, K = 2, 6, 5, 64, 128, 8, 2
    X = torch.randn((B, H, Wi, Cin)).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin)).to(BF16)
    Yc = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    xp = torch.nn.functional.pad(X.float(), (0, 0, 1, 1, 1, 1))
    cols = torch.stack([xp[:, kh:kh + H, kw:kw + Wi, :] for kh in range(3) for kw in range(3)], dim=3)
    Xcol = cols.reshape(B * H * Wi, 9 * Cin).to(BF16)
    Yl = run_linear(dev, Xcol, W, G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.equal(Yc.reshape(-1, Cout).view(torch.int32), Yl.view(torch.int32))


# ---------------------------------------------------------------------------
# 3x3 convolutions (stride 1, padding 1, 256 input channels or more) from halo
# copies: one copy of the input halo per tile and 64-channel chunk, every tap
# reading it at a row offset; 56, 28 and 14 wide images, a ragged last row
# block, a 62-wide image (64-row halo lines), 4-6 chunks per tile (the ring of
# halo buffers wraps within and across tiles), N tiles of 64, 128 and 256.
# Every output checked.
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("B,H,Wi,Cin,Cout", [(1, 56, 56, 256, 64), (2, 28, 28, 256, 128), (9, 14, 14, 256, 256),
                                             (2, 30, 30, 320, 96), (1, 17, 62, 256, 64), (3, 20, 20, 384, 192)])
def test_halo_conv3x3(dev, B, H, Wi, Cin, Cout):
    G, K = 8, 2
    g = torch.Generator().manual_seed(B * 53 + H + Cin + Cout)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, 3, 3, (1, 1), (1, 1))
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, f"halo conv B={B} {H}x{Wi} {Cin}->{Cout}")


# 64 -> 64 (and narrower) 3x3 layers: halo copies with the nine weight tiles
# resident in the stages, copied for each CTA's first tile only; more tiles than
# SMs (later tiles reuse the weights), a ragged 48-channel N tile, a ragged last
# row block.  Every output checked.
@pytest.mark.parametrize("B,H,Wi,Cout", [(100, 14, 14, 64), (170, 9, 9, 64), (3, 23, 31, 48)])
def test_halo_conv3x3_resident_weights(dev, B, H, Wi, Cout):
    Cin, G, K = 64, 8, 2
    g = torch.Generator().manual_seed(B * 7 + H + Cout)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, 3, 3, (1, 1), (1, 1))
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, f"resident halo conv B={B} {H}x{Wi} 64->{Cout}")


def test_halo_conv3x3_wide_tiles(dev):
    """Enough tiles that the 256-wide N tile wins (three stages of 32 KB beside
    the two halo buffers); sampled outputs of the first and last images."""
    B, H, Cin, Cout, G, K = 64, 14, 256, 512, 8, 2
    g = torch.Generator().manual_seed(4242)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    _, _, Wd, mask = oracle_reference(W, G, K)
    per = H * H
    for b in (0, B - 1):
        pts = np.unique(np.concatenate([np.arange(40), np.arange(per - 40, per),
                                        np.random.default_rng(b).choice(per, size=48)]))
        Yo, S = oracle.conv2d(f64(X[b:b + 1]), Wd, mask, 3, 3, (1, 1), (1, 1), pts=pts)
        Yg = f64(Y[b].reshape(-1, Cout)[torch.from_numpy(pts).to(dev)])
        assert_within_tol(Yg, Yo, S, f"halo conv wide tiles image {b}")


def test_halo_conv3x3_pair_tiles_odd_row_blocks(dev):
    """Halo copies over CTA pairs (256 input channels, the 256-wide N tile wins the
    pair count): 77 images of 9 x 9 are 77 row blocks, so the last pair's odd CTA
    has none (its halo copy and output store fall wholly outside the batch).
    Every output of the first, a middle and the last two images checked."""
    B, H, Cin, Cout, G, K = 77, 9, 256, 256, 8, 2
    g = torch.Generator().manual_seed(777)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    _, _, Wd, mask = oracle_reference(W, G, K)
    for b in (0, 38, B - 2, B - 1):
        Yo, S = oracle.conv2d(f64(X[b:b + 1]), Wd, mask, 3, 3, (1, 1), (1, 1))
        assert_within_tol(f64(Y[b]).reshape(-1, Cout), Yo, S, f"halo pair conv image {b}")


def test_halo_conv3x3_pair_tiles_ragged(dev):
    """Halo copies over CTA pairs with a ragged N tile (320 = 256 + 64 output
    channels, the second pair's tile three quarters out of range) and five
    64-channel chunks per tile (the ring of halo buffers wraps within and across
    tiles); 38 images of 14 x 14 make 38 pair units, where the 256-wide tile ties
    the 64-wide one in the pair count.  Every output of four images checked."""
    B, H, Cin, Cout, G, K = 38, 14, 320, 320, 8, 2
    g = torch.Generator().manual_seed(3838)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (1, 1), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    _, _, Wd, mask = oracle_reference(W, G, K)
    for b in (0, 17, B - 2, B - 1):
        Yo, S = oracle.conv2d(f64(X[b:b + 1]), Wd, mask, 3, 3, (1, 1), (1, 1))
        assert_within_tol(f64(Y[b]).reshape(-1, Cout), Yo, S, f"ragged halo pair conv image {b}")


# ---------------------------------------------------------------------------
# CTA-pair tiles (tcgen05 cta_group::2): bf16 layers with at least 16 stages of
# 64 reduction indices and 256-wide N tiles run as 256-row tiles split over two
# SMs.  Sizes below make the tile-round model pick that form; checked on sampled
# outputs (first and last rows, the odd last M tile whose pair partner has no
# rows, random rows).
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("N,Cin,Cout,G,K", [(38912 + 77, 1024, 736, 8, 2), (39040, 1088, 512, 16, 4)])
def test_pair_tiles_product(dev, N, Cin, Cout, G, K):
    X, W = wl.random_small(N + Cin, "bf16", N, Cin, Cout)
    Y = run_linear(dev, X, W, G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    rows = np.unique(np.concatenate([sample_rows(N, 768, seed=N), np.arange(N - 200, N)]))
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, f"pair product {N}x{Cin}->{Cout}")


@pytest.mark.parametrize("B,H,Cin,Cout,stride", [(63, 14, 128, 256, 1), (64, 28, 128, 256, 2)])
def test_pair_tiles_conv(dev, B, H, Cin, Cout, stride):
    G, K = 8, 2
    g = torch.Generator().manual_seed(B * 31 + H)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    Y = run_conv(dev, X, W, (3, 3, (stride, stride), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    P = (H + 2 - 3) // stride + 1
    per = P * P
    _, _, Wd, mask = oracle_reference(W, G, K)
    for b in (0, B - 1):
        pts = np.unique(np.concatenate([np.arange(min(per, 64)), np.arange(per - 32, per),
                                        np.random.default_rng(b).choice(per, size=64)]))
        Yo, S = oracle.conv2d(f64(X[b:b + 1]), Wd, mask, 3, 3, (stride, stride), (1, 1), pts=pts)
        Yg = f64(Y[b].reshape(-1, Cout)[torch.from_numpy(pts).to(dev)])
        assert_within_tol(Yg, Yo, S, f"pair conv B={B} H={H} s={stride} image {b}")


# fp32 layers (the split product) with long reductions: odd M tile counts,
# ragged reductions and N tails, both N tiles, 2-D and 4-D copies, checked on
# sampled outputs (products) or every output (convolutions).
@pytest.mark.parametrize("N,Cin,Cout,G,K", [(16429, 256, 1024, 8, 2), (5000, 300, 192, 16, 4), (300, 512, 64, 4, 1)])
def test_f32split_long_reduction_product(dev, N, Cin, Cout, G, K):
    X, W = wl.random_small(N + Cin + 1, "f32", N, Cin, Cout)
    Y = run_linear(dev, X, W, G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    rows = np.unique(np.concatenate([sample_rows(N, 768, seed=N), np.arange(N - 200, N)]))
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    assert_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yo, S, f"f32split product {N}x{Cin}->{Cout}")


@pytest.mark.parametrize("B,H,Cin,Cout,stride", [(9, 14, 64, 128, 1), (8, 28, 32, 64, 2), (3, 7, 256, 256, 1)])
def test_f32split_long_reduction_conv(dev, B, H, Cin, Cout, stride):
    G, K = 8, 2
    g = torch.Generator().manual_seed(B * 37 + H + Cin)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0)
    W = torch.randn((Cout, 9 * Cin), generator=g)
    Y = run_conv(dev, X, W, (3, 3, (stride, stride), (1, 1), Cout), G, K, cci.ALGO_DENSE_TC_WS)
    assert torch.isfinite(Y).all()
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, 3, 3, (stride, stride), (1, 1))
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, f"f32split conv B={B} H={H} s={stride}")


# ---------------------------------------------------------------------------
# fused output epilogue: + bias, ReLU, fp32 or bf16 (round to nearest even)
# output, on every activation source and tile form of the workspace family
# ---------------------------------------------------------------------------
from parity_util import assert_fused_within_tol  # noqa: E402

# (N, Cin, Cout, G, K, in dtype, bias, relu, out dtype)
FUSED_PRODUCTS = [
    (300, 64, 256, 8, 2, "bf16", True, True, "bf16"),
    (300, 64, 256, 8, 2, "bf16", True, False, "f32"),
    (1000, 128, 136, 8, 2, "bf16", False, True, "bf16"),
    (517, 96, 128, 16, 4, "f32", True, True, "bf16"),
    (129, 256, 1024, 8, 2, "f32", True, False, "f32"),
    # narrow last chunks: 16, 24 and 88 (= 64 + 24) bf16 output channels, 20 fp32 ones
    (2000, 32, 16, 8, 2, "bf16", True, True, "bf16"),
    (1000, 64, 24, 8, 2, "bf16", True, False, "bf16"),
    (700, 128, 88, 8, 2, "bf16", False, True, "bf16"),
    (900, 64, 20, 4, 2, "bf16", True, True, "f32"),
]


def _bias(Cout, seed):
    return (torch.randn(Cout, generator=torch.Generator().manual_seed(seed)) * 0.5).float()


@pytest.mark.parametrize("case", FUSED_PRODUCTS, ids=lambda c: "N{}_C{}x{}_G{}K{}_{}_b{}_r{}_{}".format(*c))
def test_fused_product(dev, case):
    N, Cin, Cout, G, K, dt, use_bias, relu, od = case
    X, W = wl.random_small(N + Cout, dt, N, Cin, Cout)
    b = _bias(Cout, N) if use_bias else None
    v, i = cci.pack(W.to(dev), G, K)
    Y = cci.linear_fused(X.to(dev), v, i, Cout, G, K, bias=b.to(dev) if b is not None else None, relu=relu,
                         out_dtype=_dt(od))
    assert Y.dtype == _dt(od)
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    Yr, Sr = oracle.epilogue(Yo, S, f64(b) if b is not None else None, relu)
    assert_fused_within_tol(f64(Y), Yr, Sr, od == "bf16", str(case))
    if relu:
        assert (f64(Y) >= 0).all()


# (B, H, W, Cin, Cout, KH, KW, stride, pad, G, K, in dtype): 4-D copy, stride-2
# lattices, row gather (stride 3), fp32 input
FUSED_CONVS = [
    (3, 9, 7, 64, 64, 3, 3, (1, 1), (1, 1), 8, 2, "bf16"),
    (3, 14, 14, 256, 128, 3, 3, (1, 1), (1, 1), 8, 2, "bf16"),  # halo copies
    (2, 9, 7, 64, 128, 3, 3, (2, 2), (1, 1), 8, 2, "bf16"),
    (1, 10, 10, 64, 64, 3, 3, (3, 3), (1, 1), 8, 2, "bf16"),
    (2, 9, 7, 32, 64, 3, 3, (1, 1), (1, 1), 8, 2, "f32"),
]


@pytest.mark.parametrize("od", ["bf16", "f32"])
@pytest.mark.parametrize("case", FUSED_CONVS, ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_G{}K{}_{}".format(*c))
def test_fused_conv(dev, case, od):
    B, H, Wi, Cin, Cout, KH, KW, stride, pad, G, K, dt = case
    g = torch.Generator().manual_seed(B * 41 + Cin + Cout)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(_dt(dt))
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(_dt(dt))
    b = _bias(Cout, B + Cout)
    v, i = cci.pack(W.to(dev), G, K)
    Y = cci.conv2d_fused(X.to(dev), v, i, Cout, G, K, KH, KW, stride, pad, bias=b.to(dev), relu=True,
                         out_dtype=_dt(od))
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.conv2d(f64(X), Wd, mask, KH, KW, stride, pad)
    Yr, Sr = oracle.epilogue(Yo, S, f64(b), True)
    assert_fused_within_tol(f64(Y).reshape(-1, Cout), Yr, Sr, od == "bf16", str(case))


def test_fused_pair_tiles(dev):
    """CTA-pair tiles (long reduction, 256-wide N tile) with bias, ReLU and bf16
    output; sampled rows."""
    N, Cin, Cout, G, K = 38912 + 77, 1024, 736, 8, 2
    X, W = wl.random_small(N + 1, "bf16", N, Cin, Cout)
    b = _bias(Cout, 3)
    v, i = cci.pack(W.to(dev), G, K)
    Y = cci.linear_fused(X.to(dev), v, i, Cout, G, K, bias=b.to(dev), relu=True, out_dtype=BF16)
    rows = np.unique(np.concatenate([sample_rows(N, 512, seed=9), np.arange(N - 160, N)]))
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X[rows]), Wd, mask)
    Yr, Sr = oracle.epilogue(Yo, S, f64(b), True)
    assert_fused_within_tol(f64(Y[torch.from_numpy(rows).to(dev)]), Yr, Sr, True, "fused pair")


def test_fused_halo_pair_tiles(dev):
    """Bias, ReLU and bf16 output on halo copies over CTA pairs (256 input
    channels, two 256-wide N tiles), through the workspace family; every output of
    the first and last images."""
    B, H, Cin, Cout, G, K = 64, 14, 256, 512, 8, 2
    g = torch.Generator().manual_seed(5150)
    X = torch.randn((B, H, H, Cin), generator=g).clamp_min(0).to(BF16)
    W = torch.randn((Cout, 9 * Cin), generator=g).to(BF16)
    b = _bias(Cout, 7)
    v, i = cci.pack(W.to(dev), G, K)
    ws = cci.new_workspace(cci.ALGO_DENSE_TC_WS, BF16, Cout, 9 * Cin, dev)
    Y = cci.conv2d_fused(X.to(dev), v, i, Cout, G, K, 3, 3, (1, 1), (1, 1), bias=b.to(dev), relu=True,
                         out_dtype=BF16, workspace=ws)
    _, _, Wd, mask = oracle_reference(W, G, K)
    for img in (0, B - 1):
        Yo, S = oracle.conv2d(f64(X[img:img + 1]), Wd, mask, 3, 3, (1, 1), (1, 1))
        Yr, Sr = oracle.epilogue(Yo, S, f64(b), True)
        assert_fused_within_tol(f64(Y[img]).reshape(-1, Cout), Yr, Sr, True, f"fused halo pair image {img}")


def test_fused_identity_equals_plain_product(dev):
    """No bias, no ReLU, fp32 output: bit for bit the plain product of the family
    AUTO picks (the binding passes both calls the workspace AUTO asks for), and,
    with no workspace, of the fused family."""
    for G, K in ((8, 2), (16, 8)):
        N, Cin, Cout = 700, 128, 256
        X, W = wl.random_small(5, "bf16", N, Cin, Cout)
        Xd = X.to(dev)
        v, i = cci.pack(W.to(dev), G, K)
        Yf = cci.linear_fused(Xd, v, i, Cout, G, K)
        Yp = cci.linear(Xd, v, i, Cout, G, K)
        assert torch.equal(Yf.view(torch.int32), Yp.view(torch.int32))
    G, K = 8, 2
    v, i = cci.pack(W.to(dev), G, K)
    Yf = torch.empty((N, Cout), device=dev)
    code = cci.lib().cci_linear_fused(Xd.data_ptr(), cci.BF16, N, Cin, v.data_ptr(), i.data_ptr(), Cout, G, K,
                                      None, 0, cci.F32, Yf.data_ptr(), None, None, 0,
                                      torch.cuda.current_stream(dev).cuda_stream)
    assert code == 0
    Yp = cci.linear(Xd, v, i, Cout, G, K, algo=cci.ALGO_DENSE_TC)
    assert torch.equal(Yf.view(torch.int32), Yp.view(torch.int32))


# ---------------------------------------------------------------------------
# allocation statistics of packing (Eq. 1 measured): exact counts against the
# oracle, and the counted ratio against the closed form on independent zeros
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("Cout,R,G,K,Ps", [(64, 33, 8, 2, 0.75), (48, 1000, 16, 4, 0.5), (1024, 4096, 8, 2, 0.75),
                                           (4, 7, 4, 1, 0.3), (512, 96, 32, 8, 0.9),
                                           (90, 21, 3, 1, 0.4), (128, 40, 64, 16, 0.5)])
def test_pack_stats_exact(dev, dtype, Cout, R, G, K, Ps):
    rng = np.random.default_rng(Cout + R + G)
    W = rng.standard_normal((Cout, R)).astype(np.float32)
    W[rng.random((Cout, R)) < Ps] = 0
    W[-1, : min(R, 6)] = -0.0
    Wt = torch.from_numpy(W).to(_dt(dtype))
    counts = cci.pack_stats(Wt.to(dev), G, K)
    got = counts.cpu().tolist()
    assert got == list(oracle.pack_stats(f64(Wt), G, K))
    cci.pack_stats(Wt.to(dev), G, K, counts=counts)  # accumulates
    assert counts.cpu().tolist() == [2 * got[0], 2 * got[1]]


@pytest.mark.parametrize("G,Ps", [(4, 0.5), (8, 0.75), (16, 0.875), (64, 0.75), (256, 0.9375)])
def test_pack_stats_estimates_eq1(dev, G, Ps):
    """Independent zeros with probability Ps, K = G(1 - Ps): the GPU-counted
    dropped fraction is within 5 standard errors of Eq. 1."""
    K = int(round(G * (1 - Ps)))
    g = torch.Generator(device="cuda").manual_seed(G)
    Cout, R = 4096, 8192
    W = torch.randn((Cout, R), generator=g, device=dev)
    W[torch.rand((Cout, R), generator=g, device=dev) < Ps] = 0
    nz, dropped = cci.pack_stats(W, G, K).cpu().tolist()
    groups = (Cout // G) * R
    est = dropped / nz
    pd = oracle.allocation_error(G, Ps)
    # per group the overflow is at most G - K; its variance is bounded by E[over] * (G - K)
    se = np.sqrt(pd * K * (G - K) / groups) / K
    assert abs(est - pd) < 5 * se + 1e-9, (est, pd, se)


# ---------------------------------------------------------------------------
# the same tensor-core GEMM on dense (unpruned) weights: the reference line of
# what the sparsity buys
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("N,Cin,Cout", [(300, 64, 256), (129, 72, 40), (1000, 256, 1024), (2048, 512, 512)])
def test_dense_linear_tc(dev, dtype, N, Cin, Cout):
    X, W = wl.random_small(N + Cin + 1, dtype, N, Cin, Cout)
    Y = torch.full((N, Cout), float("nan"), device=dev)
    st = cci.new_status(dev)
    cci.dense_linear_tc(X.to(dev), cci.dense_planes(W.to(dev)), Cout, out=Y, status=st)
    assert cci.read_status(st) == 0
    Yo, S = oracle.linear(f64(X), f64(W), np.ones((Cout, Cin), dtype=bool))
    assert_within_tol(f64(Y), Yo, S, f"dense {dtype} {N}x{Cin}->{Cout}")


@pytest.mark.parametrize("case", [(2, 14, 14, 64, 128, 3, 3, 1, 1, "bf16"), (3, 9, 9, 32, 64, 3, 3, 2, 1, "bf16"),
                                  (2, 8, 8, 16, 32, 1, 1, 1, 0, "f32")],
                         ids=lambda c: "B{}_{}x{}_{}to{}_k{}x{}_s{}_p{}_{}".format(*c))
def test_dense_conv2d_tc(dev, case):
    B, H, Wi, Cin, Cout, KH, KW, s, p, dtype = case
    g = torch.Generator().manual_seed(B + Cin)
    X = torch.randn((B, H, Wi, Cin), generator=g).clamp_min(0).to(_dt(dtype))
    W = torch.randn((Cout, KH * KW * Cin), generator=g).to(_dt(dtype))
    st = cci.new_status(dev)
    Y = cci.dense_conv2d_tc(X.to(dev), cci.dense_planes(W.to(dev)), Cout, KH, KW, (s, s), (p, p), status=st)
    assert cci.read_status(st) == 0
    Yo, S = oracle.conv2d(f64(X), f64(W), np.ones(W.shape, dtype=bool), KH, KW, (s, s), (p, p))
    assert_within_tol(f64(Y).reshape(-1, Cout), Yo, S, str(case))
