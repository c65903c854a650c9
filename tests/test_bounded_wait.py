"""The bounded waits of the tensor-core kernels, exercised through cci_wait_probe.

Every copy and MMA wait in those kernels gives up after about a second, records
CCI_ERR_TIMEOUT in the caller's status word and lets the kernel return.  Here a
wait is made to run out the sanctioned way -- on a barrier that nothing else
arrives on -- and the host reads the status; the same context then runs a
product that must still match the oracle.  Nothing faults, traps or hangs.
"""
import time

import pytest
import torch

import oracle
import paper_1910_11971_gb300 as cci
from paper_1910_11971_gb300 import build as cci_build
from paper_1910_11971_gb300 import workloads as wl
from parity_util import assert_within_tol, f64, oracle_reference

TIMEOUT = 8  # CCI_ERR_TIMEOUT


def test_probe_needs_a_status_word():
    cci_build.build()
    assert cci.lib().cci_wait_probe(None, 0, None) == 1  # CCI_ERR_NULL, before any launch


@pytest.mark.gpu
def test_wait_with_its_arrival_returns_cleanly():
    cci_build.build()
    dev = torch.device("cuda:0")
    st = cci.new_status(dev)
    t0 = time.perf_counter()
    assert cci.lib().cci_wait_probe(st.data_ptr(), 1, torch.cuda.current_stream(dev).cuda_stream) == 0
    assert cci.read_status(st) == 0
    assert time.perf_counter() - t0 < 0.5


@pytest.mark.gpu
def test_expired_wait_reports_timeout_and_the_context_stays_usable():
    cci_build.build()
    dev = torch.device("cuda:0")
    st = cci.new_status(dev)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    assert cci.lib().cci_wait_probe(st.data_ptr(), 0, torch.cuda.current_stream(dev).cuda_stream) == 0
    code = cci.read_status(st)  # synchronises
    waited = time.perf_counter() - t0
    assert code == TIMEOUT
    assert int(st.item()) == 1 << TIMEOUT
    assert 0.2 < waited < 30.0, waited  # ~2^31 SM cycles
    # the same context goes on computing correctly
    X, W = wl.random_small(5, "f32", 300, 64, 256)
    v, i = cci.pack(W.to(dev), 8, 2)
    st2 = cci.new_status(dev)
    Y = cci.linear(X.to(dev), v, i, 256, 8, 2, status=st2)
    assert cci.read_status(st2) == 0
    _, _, Wd, mask = oracle_reference(W, 8, 2)
    Yo, S = oracle.linear(f64(X), Wd, mask)
    assert_within_tol(f64(Y), Yo, S, "product after an expired wait")
