"""The static-scratch product, cci_linear_dense_tc_static.

It serves callers that cannot allocate device memory (a plug-in inside a host
framework that owns all device memory, a serving loop that forbids allocation
after start-up): instead of a caller workspace, the dense weights go to a static
device array inside the library.  Its output must match the workspace product
(cci_linear_ws with CCI_ALGO_DENSE_TC_WS) on the same inputs, within the parity
tolerance, on three calls in a row with different layers (the array keeps the
last call's contents, so a stale region must never leak into the next result),
and on a layer whose dense weights fill the array to its last byte.
This file is collected last on purpose.
"""
import pytest
import torch

import oracle
import paper_1910_11971_gb300 as cci
from paper_1910_11971_gb300 import build as cci_build
from paper_1910_11971_gb300 import workloads as wl
from parity_util import assert_within_tol, f64, oracle_reference

STATIC_BYTES = 16 * 1024 * 1024
FAKE = 0x10000


def call_static(X, v, i, Cout, G, K, Y, status):
    return cci.lib().cci_linear_dense_tc_static(
        X.data_ptr(), cci.BF16, X.shape[0], X.shape[1], v.data_ptr(), i.data_ptr(), Cout, G, K,
        Y.data_ptr(), status.data_ptr(), torch.cuda.current_stream().cuda_stream)


def test_static_scratch_rejects_layers_over_the_limit():
    cci_build.build()
    lib = cci.lib()
    # 4096 x 4096 bf16 dense weights are 32 MiB > 16 MiB: rejected before any launch
    assert lib.cci_linear_dense_tc_static(FAKE, cci.BF16, 16, 4096, FAKE, FAKE, 4096, 8, 2, FAKE,
                                          None, None) == 11
    assert lib.cci_linear_dense_tc_static(FAKE, cci.F32, 16, 64, FAKE, FAKE, 256, 8, 2, FAKE,
                                          None, None) != 0  # fp32 has no dense tensor-core kernel
    assert 4096 * 2048 * 2 == STATIC_BYTES
    # one 8-channel step over the limit: 4096 x 2056 bf16 is rejected
    assert lib.cci_linear_dense_tc_static(FAKE, cci.BF16, 16, 2056, FAKE, FAKE, 4096, 8, 2, FAKE,
                                          None, None) == 11
    # a shape whose Cout * Cin overflows is a shape error, not a size error
    assert lib.cci_linear_dense_tc_static(FAKE, cci.BF16, 16, 1 << 40, FAKE, FAKE, 1 << 40, 8, 2, FAKE,
                                          None, None) == 2


@pytest.mark.gpu
def test_static_scratch_product_matches_workspace_product():
    cci_build.build()
    dev = torch.device("cuda:0")
    # three calls in a row: a small layer (32 KiB of dense weights), then one that
    # covers 32x more of the array (1 MiB), then the first again (the array then
    # holds the larger layer's weights beyond the small layer's region)
    layers = [(300, 64, 256, 8, 2, 11), (1000, 512, 1024, 16, 4, 12), (300, 64, 256, 8, 2, 13)]
    for N, Cin, Cout, G, K, seed in layers:
        X, W = wl.random_small(seed, "bf16", N, Cin, Cout)
        Xd = X.to(dev)
        v, i = cci.pack(W.to(dev), G, K)
        Ys = torch.full((N, Cout), float("nan"), device=dev)
        st = cci.new_status(dev)
        assert call_static(Xd, v, i, Cout, G, K, Ys, st) == 0
        Yw = cci.linear(Xd, v, i, Cout, G, K, algo=cci.ALGO_DENSE_TC_WS)
        assert cci.read_status(st) == 0
        _, _, Wd, mask = oracle_reference(W, G, K)
        Yo, S = oracle.linear(f64(X), Wd, mask)
        assert_within_tol(f64(Ys), f64(Yw), S, f"static vs workspace {N}x{Cin}->{Cout}")
        assert_within_tol(f64(Ys), Yo, S, f"static vs oracle {N}x{Cin}->{Cout}")


@pytest.mark.gpu
def test_static_scratch_at_the_limit():
    """4096 output channels x 2048 inputs in bf16: the dense weights fill the 16 MiB
    array exactly, so the decompression writes and the GEMM's weight copies reach
    its last bytes (the last output channels read them).  Every output is compared
    with the workspace product and with the oracle."""
    cci_build.build()
    dev = torch.device("cuda:0")
    N, Cin, Cout, G, K = 200, 2048, 4096, 8, 2
    assert Cout * Cin * 2 == STATIC_BYTES
    X, W = wl.random_small(21, "bf16", N, Cin, Cout)
    Xd = X.to(dev)
    v, i = cci.pack(W.to(dev), G, K)
    Ys = torch.full((N, Cout), float("nan"), device=dev)
    st = cci.new_status(dev)
    assert call_static(Xd, v, i, Cout, G, K, Ys, st) == 0
    Yw = cci.linear(Xd, v, i, Cout, G, K, algo=cci.ALGO_DENSE_TC_WS)
    assert cci.read_status(st) == 0
    _, _, Wd, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Ys), f64(Yw), S, "static vs workspace at the limit")
    assert_within_tol(f64(Ys), Yo, S, "static vs oracle at the limit")
