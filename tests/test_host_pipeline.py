"""cci_linear_host: the product with X and Y in host memory, column chunks
copied in, multiplied and copied out on three streams.

CPU: argument checks return before anything is enqueued, and the device buffer
size is the workspace plus two staging slots per direction.  GPU: the result
equals the device-resident product (cci_linear_ws, dense tensor-core family)
bit for bit, and the oracle within the product's tolerance, over ragged chunk
counts, both dtypes, pinned and pageable host memory, and with the copies on
their own streams or on the compute stream.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_1910_11971_gb300 as cci
from paper_1910_11971_gb300 import build as cci_build
from paper_1910_11971_gb300 import workloads as wl
from parity_util import assert_within_tol, f64, oracle_reference

FAKE = 0x10000  # an aligned address that is never dereferenced by the argument checks


def _r256(b):
    return (b + 255) // 256 * 256


@pytest.fixture(scope="module")
def lib():
    cci_build.build()
    return cci.lib()


def call(lib, N=16, Cin=64, Cout=256, G=8, K=2, dtype=cci.F32, chunk=128, buf=FAKE, nbytes=1 << 40,
         X=FAKE, Y=FAKE):
    return lib.cci_linear_host(X, dtype, N, Cin, FAKE, FAKE, Cout, G, K, Y, chunk, buf, nbytes, None, None,
                               None, None)


def test_buffer_size(lib):
    # fp32: workspace Cout*Cin*8, slots chunk*Cin*4 in and chunk*Cout*4 out, two of each
    assert lib.cci_linear_host_buffer_size(cci.F32, 256, 1024, 12544) == \
        _r256(1024 * 256 * 8) + 2 * (_r256(12544 * 256 * 4) + _r256(12544 * 1024 * 4))
    assert lib.cci_linear_host_buffer_size(cci.BF16, 72, 40, 100) == \
        _r256(40 * 72 * 2) + 2 * (_r256(100 * 72 * 2) + _r256(100 * 40 * 4))
    assert lib.cci_linear_host_buffer_size(cci.F32, 64, 64, 0) == 0
    assert lib.cci_linear_host_buffer_size(7, 64, 64, 128) == 0


def test_rejects_before_any_launch(lib):
    need = lib.cci_linear_host_buffer_size(cci.F32, 64, 256, 128)
    assert call(lib, chunk=0) == 2                     # CCI_ERR_SHAPE
    assert call(lib, nbytes=need - 1) == 11            # CCI_ERR_WORKSPACE: short
    assert call(lib, buf=None) == 11                   # missing
    assert call(lib, buf=FAKE + 16) == 11              # not 256-byte aligned
    assert call(lib, G=8, K=8) == 9                    # CCI_ERR_UNSUPPORTED: no dense kernel for K = G
    assert call(lib, Cin=66) == 9                      # fp32 needs Cin % 4 == 0
    assert call(lib, dtype=cci.BF16, Cin=68) == 9      # bf16 needs Cin % 8 == 0
    assert call(lib, Cout=250) == 3                    # CCI_ERR_GROUP: Cout % G
    assert call(lib, dtype=5) == 4                     # CCI_ERR_DTYPE
    assert call(lib, X=None) == 1                      # CCI_ERR_NULL
    assert call(lib, N=-1) == 2


def test_empty_input_enqueues_nothing(lib):
    assert call(lib, N=0, nbytes=lib.cci_linear_host_buffer_size(cci.F32, 64, 256, 128)) == 0


CASES = [  # (dtype, N, Cin, Cout, G, K, chunk)
    ("f32", 300, 64, 256, 8, 2, 128),      # three chunks, the last ragged (44 columns)
    ("f32", 1000, 256, 512, 8, 2, 384),    # chunks of 3 tiles, ragged tail
    ("f32", 100, 64, 64, 4, 2, 512),       # one chunk larger than N
    ("bf16", 1000, 128, 256, 16, 4, 256),  # four chunks, the last ragged
    ("bf16", 129, 64, 128, 8, 1, 1),       # one column per chunk (129 chunks)
]


@pytest.mark.gpu
@pytest.mark.parametrize("dtype,N,Cin,Cout,G,K,chunk", CASES)
@pytest.mark.parametrize("mode", ["streams", "one_stream", "pageable"])
def test_host_product_matches_device_product(dtype, N, Cin, Cout, G, K, chunk, mode):
    cci_build.build()
    dev = torch.device("cuda:0")
    X, W = wl.random_small(N * 7 + Cin, dtype, N, Cin, Cout)
    Wd = W.to(dev)
    v, i = cci.pack(Wd, G, K)
    st = cci.new_status(dev)
    Xh = X.contiguous() if mode == "pageable" else X.contiguous().pin_memory()
    Yh = torch.full((N, Cout), float("nan"), dtype=torch.float32)
    if mode != "pageable":
        Yh = Yh.pin_memory()
    if mode == "one_stream":
        # the copies on the compute stream (NULL copy streams), through the C ABI
        buf = cci.host_buffer(Xh.dtype, Cin, Cout, chunk, dev)
        code = cci.lib().cci_linear_host(Xh.data_ptr(), cci._dtype_code(Xh), N, Cin, v.data_ptr(), i.data_ptr(),
                                         Cout, G, K, Yh.data_ptr(), chunk, buf.data_ptr(), buf.numel(),
                                         st.data_ptr(), torch.cuda.current_stream(dev).cuda_stream, None, None)
        assert code == 0
    else:
        cci.linear_host(Xh, v, i, Cout, G, K, out=Yh, status=st, chunk=chunk)
    torch.cuda.current_stream(dev).synchronize()
    assert cci.read_status(st) == 0
    Yd = cci.linear(X.to(dev), v, i, Cout, G, K, algo=cci.ALGO_AUTO).cpu()
    same = Yh.view(torch.int32) == Yd.view(torch.int32)
    assert bool(same.all()), f"{int((~same).sum())} outputs differ from the device-resident product"
    _, _, Wo, mask = oracle_reference(W, G, K)
    Yo, S = oracle.linear(f64(X), Wo, mask)
    assert_within_tol(f64(Yh), Yo, S, f"host product {dtype} N={N} chunk={chunk} {mode}")


@pytest.mark.gpu
def test_host_product_orders_after_prior_work_and_reuses_the_buffer():
    """Two calls in a row on one buffer, the second on different inputs, each
    right after the pack that produces its weights on the same stream."""
    cci_build.build()
    dev = torch.device("cuda:0")
    N, Cin, Cout, G, K, chunk = 700, 64, 256, 8, 2, 256
    buf = cci.host_buffer(torch.float32, Cin, Cout, chunk, dev)
    for seed in (1, 2):
        X, W = wl.random_small(seed, "f32", N, Cin, Cout)
        v, i = cci.pack(W.to(dev), G, K)  # enqueued on the current stream just before
        Yh = cci.linear_host(X.pin_memory(), v, i, Cout, G, K, chunk=chunk, buffer=buf)
        torch.cuda.current_stream(dev).synchronize()
        _, _, Wo, mask = oracle_reference(W, G, K)
        Yo, S = oracle.linear(f64(X), Wo, mask)
        assert_within_tol(f64(Yh), Yo, S, f"call {seed}")


@pytest.mark.gpu
def test_host_product_bottleneck_full():
    """The benchmark's end-to-end call at full size (N = 100352, 256 -> 1024, G = 8,
    K = 2, fp32, 12544-column chunks): every output equals the device-resident
    product, and sampled rows (tile and chunk edges, the tail, random ones) are
    within tolerance of the oracle."""
    from parity_util import sample_rows
    cci_build.build()
    dev = torch.device("cuda:0")
    case = wl.BOTTLENECK_1X1
    X, W = wl.linear_inputs(case)
    v, i = cci.pack(W.to(dev), case.G, case.K)
    chunk = cci.host_chunk(case.N)
    assert chunk == 12544
    st = cci.new_status(dev)
    Yh = cci.linear_host(X.pin_memory(), v, i, case.Cout, case.G, case.K, status=st, chunk=chunk)
    torch.cuda.current_stream(dev).synchronize()
    assert cci.read_status(st) == 0
    Yd = cci.linear(X.to(dev), v, i, case.Cout, case.G, case.K, algo=cci.ALGO_AUTO).cpu()
    assert bool((Yh.view(torch.int32) == Yd.view(torch.int32)).all())
    edges = np.concatenate([np.arange(c * chunk - 2, c * chunk + 2) for c in range(1, case.N // chunk)])
    rows = np.unique(np.concatenate([sample_rows(case.N, 1024, seed=5), edges]))
    _, _, Wo, mask = oracle_reference(W, case.G, case.K)
    Yo, S = oracle.linear(f64(X[rows]), Wo, mask)
    assert_within_tol(f64(Yh[torch.from_numpy(rows)]), Yo, S, "bottleneck_1x1 through cci_linear_host")
