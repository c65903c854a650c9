"""The C ABI without a GPU: libcci.so builds, loads, exports every entry point
that include/cci.h declares, and rejects bad arguments with the documented
status before anything is enqueued (these paths never touch the device)."""
import ctypes
import os
import re

import pytest

import paper_1910_11971_gb300 as cci
from paper_1910_11971_gb300 import build as cci_build

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cci.h")

OK, NULL, SHAPE, GROUP, DTYPE, ALIGN, VALUE, CUDA, TIMEOUT, UNSUP, INDEX = range(11)
FAKE = 0x10000  # a 256-byte-aligned non-null address; never dereferenced on these paths


@pytest.fixture(scope="module")
def lib():
    cci_build.build()
    return cci.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(cci_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("cci_pack", "cci_linear", "cci_conv2d", "cci_status_string"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    missing = [n for n in declared_functions() if not hasattr(lib, n)]
    assert not missing
    assert set(declared_functions()) == set(cci.SIGNATURES)


def test_version_and_strings(lib):
    assert lib.cci_version() >= 10000
    for code in range(11):
        assert lib.cci_status_string(code)
    assert lib.cci_status_string(OK) == b"ok"


def test_decode_device_status(lib):
    assert cci.decode_status(0) == OK
    assert cci.decode_status(1 << INDEX) == INDEX
    assert cci.decode_status((1 << INDEX) | (1 << VALUE)) == VALUE
    assert cci.decode_status(1 << TIMEOUT) == TIMEOUT


def linear(lib, X=FAKE, dt=0, N=16, Cin=16, V=FAKE, I=FAKE, Cout=16, G=8, K=2, Y=FAKE, algo=0):
    return lib.cci_linear_ex(X, dt, N, Cin, V, I, Cout, G, K, Y, None, algo, None)


def conv(lib, X=FAKE, dt=1, B=1, H=4, W=4, Cin=8, V=FAKE, I=FAKE, Cout=8, KH=3, KW=3, sh=1, sw=1,
         ph=1, pw=1, G=8, K=2, Y=FAKE, algo=0):
    return lib.cci_conv2d_ex(X, dt, B, H, W, Cin, V, I, Cout, KH, KW, sh, sw, ph, pw, G, K, Y, None,
                             algo, None)


def test_linear_rejects(lib):
    assert linear(lib, X=None) == NULL
    assert linear(lib, Y=None) == NULL
    assert linear(lib, V=None) == NULL
    assert linear(lib, I=None) == NULL
    assert linear(lib, dt=7) == DTYPE
    assert linear(lib, N=-1) == SHAPE
    assert linear(lib, Cin=0) == SHAPE
    assert linear(lib, Cout=0) == SHAPE
    assert linear(lib, G=0) == GROUP
    assert linear(lib, G=257, Cout=257) == GROUP
    assert linear(lib, K=0) == GROUP
    assert linear(lib, K=9) == GROUP
    assert linear(lib, Cout=12) == GROUP  # 12 % 8
    assert linear(lib, X=FAKE + 2) == ALIGN  # fp32 needs 4-byte alignment
    assert linear(lib, Y=FAKE + 2) == ALIGN
    assert linear(lib, N=1 << 40, Cout=1 << 30) == SHAPE  # N*Cout overflows the limit


def test_empty_input_is_ok_without_device(lib):
    # N = 0 enqueues nothing, so it succeeds even with no GPU (and NULL X / Y)
    assert linear(lib, N=0, X=None, Y=None) == OK
    assert conv(lib, B=0, X=None, Y=None) == OK


def test_conv_rejects(lib):
    assert conv(lib, H=0) == SHAPE
    assert conv(lib, KH=0) == SHAPE
    assert conv(lib, sh=0) == SHAPE
    assert conv(lib, ph=-1) == SHAPE
    assert conv(lib, H=2, KH=5, ph=1) == SHAPE  # no output row
    assert conv(lib, dt=3) == DTYPE
    assert conv(lib, G=3) == GROUP
    assert conv(lib, X=FAKE + 1) == ALIGN  # bf16 needs 2-byte alignment
    assert conv(lib, I=None) == NULL


def test_pack_rejects(lib):
    p = lib.cci_pack
    assert p(None, 0, 8, 4, 4, 2, FAKE, FAKE, None, None) == NULL
    assert p(FAKE, 0, 8, 4, 4, 2, None, FAKE, None, None) == NULL
    assert p(FAKE, 2, 8, 4, 4, 2, FAKE, FAKE, None, None) == DTYPE
    assert p(FAKE, 0, 0, 4, 4, 2, FAKE, FAKE, None, None) == SHAPE
    assert p(FAKE, 0, 8, 0, 4, 2, FAKE, FAKE, None, None) == SHAPE
    assert p(FAKE, 0, 8, 4, 3, 2, FAKE, FAKE, None, None) == GROUP
    assert p(FAKE, 0, 8, 4, 4, 5, FAKE, FAKE, None, None) == GROUP
    assert p(FAKE + 2, 0, 8, 4, 4, 2, FAKE, FAKE, None, None) == ALIGN


def test_algo_dense_tc_names(lib):
    import torch
    assert cci.kernel_name(torch.float32, 16, 16, 16, 8, 2, cci.ALGO_DENSE_TC) == ""  # bf16 only
    assert cci.kernel_name(torch.bfloat16, 16, 16, 16, 8, 2, cci.ALGO_DENSE_TC) == "dense_tc_fused_bf16_G8_K2"
    assert cci.kernel_name(torch.bfloat16, 16, 16, 64, 32, 8, cci.ALGO_DENSE_TC) == "dense_tc_fused_bf16_G32_K8"
    assert cci.kernel_name(torch.bfloat16, 16, 16, 64, 32, 16, cci.ALGO_DENSE_TC) == ""  # K = 16: no expansion
    assert cci.kernel_name(torch.bfloat16, 12, 12, 16, 8, 2, cci.ALGO_DENSE_TC) == ""  # Cin % 8
    assert cci.kernel_name(torch.bfloat16, 16, 16, 24, 8, 3, cci.ALGO_DENSE_TC) == ""  # K not a power of 2
    assert cci.kernel_name(torch.bfloat16, 24, 24, 16, 8, 1, cci.ALGO_DENSE_TC) == ""  # R * K % 16
    assert cci.kernel_name(torch.bfloat16, 64, 576, 64, 8, 2, cci.ALGO_DENSE_TC) == "dense_tc_fused_bf16_G8_K2"
    assert cci.kernel_name(torch.bfloat16, 32, 288, 64, 8, 2, cci.ALGO_DENSE_TC) == ""  # conv, Cin % 64
    # AUTO (given the workspace it asks for): a tensor-core family for these layers;
    # the workspace one for K = 8
    assert cci.kernel_name(torch.bfloat16, 16, 16, 16, 8, 2) in ("dense_tc_fused_bf16_G8_K2", "dense_tc_ws_bf16_G8_K2")
    assert cci.kernel_name(torch.bfloat16, 16, 16, 64, 32, 8) == "dense_tc_ws_bf16_G32_K8"
    # fp32: the workspace family (tf32 hi*hi plus bf16 cross terms) with a workspace; CUDA-core kernels without one
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 2) == "dense_tc_ws_f32split_G8_K2"


def test_kernel_names(lib):
    import torch
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 2, cci.ALGO_REGTILE).startswith("regtile_float_G8_K2_")
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 2, cci.ALGO_EXPAND).startswith("expand_float_G8_K2_")
    assert cci.kernel_name(torch.bfloat16, 128, 1152, 128, 16, 4, cci.ALGO_REGTILE).startswith("regtile_uint16_t_G16_K4")
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 2) != ""
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 3) == "generic_f32"  # no tile for K=3
    assert cci.kernel_name(torch.bfloat16, 12, 12, 16, 8, 2) == "generic_bf16"  # Cin % 8 != 0
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 3, cci.ALGO_REGTILE) == ""
    assert cci.kernel_name(torch.float32, 256, 256, 1024, 8, 2, cci.ALGO_GENERIC) == "generic_f32"


def test_workspace_rules(lib):
    import torch
    ws = cci.ALGO_DENSE_TC_WS
    assert cci.workspace_size(ws, torch.bfloat16, 256, 64) == 256 * 64 * 2
    assert cci.workspace_size(cci.ALGO_EXPAND, torch.bfloat16, 256, 64) == 0
    assert cci.workspace_size(cci.ALGO_AUTO, torch.float32, 256, 64) == 256 * 64 * 8
    assert cci.workspace_size(ws, torch.float32, 256, 64) == 256 * 64 * 8
    assert cci.kernel_name(torch.float32, 64, 64, 256, 8, 2, ws) == "dense_tc_ws_f32split_G8_K2"
    assert cci.kernel_name(torch.float32, 64, 64, 256, 8, 2, cci.ALGO_DENSE_TC) == ""
    assert cci.workspace_size(cci.ALGO_AUTO, torch.bfloat16, 256, 64) == 256 * 64 * 2
    # the family needs a workspace: rejected before any launch (no device needed)
    assert linear(lib, dt=1, algo=ws) == 11
    assert lib.cci_linear_ws(FAKE, 1, 16, 16, FAKE, FAKE, 16, 8, 2, FAKE, None, ws, FAKE, 16, None) == 11
    assert lib.cci_linear_ws(FAKE, 1, 16, 16, FAKE, FAKE, 16, 8, 2, FAKE, None, ws, FAKE + 8, 4096, None) == 11
    assert cci.kernel_name(torch.bfloat16, 64, 64, 256, 8, 2, ws) == "dense_tc_ws_bf16_G8_K2"
    assert cci.kernel_name(torch.bfloat16, 8, 36, 256, 8, 2, ws) == ""  # R % 8 != 0
    # fp32: plane 0 [Cout][R] of 4 bytes, plane 1 [Cout][ceil(R / 32) * 64] of 2 bytes
    assert cci.workspace_size(ws, torch.float32, 256, 72) == 256 * (72 * 4 + 3 * 128)


def test_dense_planes_rejects(lib):
    # argument checks run before any device call
    need = 64 * (40 * 4 + 2 * 128)
    assert lib.cci_dense_planes(FAKE, 0, 64, 40, FAKE, need - 1, None) == 11  # CCI_ERR_WORKSPACE
    assert lib.cci_dense_planes(FAKE, 0, 64, 40, None, need, None) == 1       # CCI_ERR_NULL
    assert lib.cci_dense_planes(FAKE + 8, 0, 64, 40, FAKE, need, None) == 5   # CCI_ERR_ALIGN (pointer)
    assert lib.cci_dense_planes(FAKE, 0, 64, 42, FAKE, 10**9, None) == 5      # CCI_ERR_ALIGN (R % 4)
    assert lib.cci_dense_planes(FAKE, 1, 64, 36, FAKE, 10**9, None) == 5      # bf16: R % 8
    assert lib.cci_dense_planes(FAKE, 0, 0, 40, FAKE, need, None) == 2        # CCI_ERR_SHAPE
    assert lib.cci_dense_planes(FAKE, 7, 64, 40, FAKE, need, None) == 4       # CCI_ERR_DTYPE


def test_fma_probe_rejects(lib):
    assert lib.cci_fma_probe(None, 1, 32, 1, None) == NULL
    assert lib.cci_fma_probe(FAKE, 0, 32, 1, None) == SHAPE
    assert lib.cci_fma_probe(FAKE, 1, 2048, 1, None) == SHAPE


def test_binding_fails_loudly_without_library(monkeypatch, tmp_path):
    monkeypatch.setattr(cci, "_lib", None)
    monkeypatch.setattr(cci, "LIB_PATH", str(tmp_path / "missing.so"))
    with pytest.raises(RuntimeError, match="not built"):
        cci.lib()


def fused(lib, X=FAKE, dt=1, N=16, Cin=64, V=FAKE, I=FAKE, Cout=64, G=8, K=2, bias=None, relu=1, od=1,
          Y=FAKE, ws=FAKE, wsb=1 << 20):
    return lib.cci_linear_fused(X, dt, N, Cin, V, I, Cout, G, K, bias, relu, od, Y, None, ws, wsb, None)


def test_fused_rejects(lib):
    """The fused epilogue (bias, ReLU, bf16 output) exists on the workspace
    tensor-core family only; every argument error is returned before a launch."""
    assert fused(lib, od=5) == DTYPE
    assert fused(lib, dt=5) == DTYPE
    assert fused(lib, V=None) == NULL
    assert fused(lib, Cout=60) == GROUP                   # Cout % G
    assert fused(lib, G=64, Cout=64) == UNSUP             # G without a dense tensor-core kernel
    assert fused(lib, G=4, K=2, Cout=68) == UNSUP         # bf16 rows need Cout % 8 == 0
    assert fused(lib, bias=FAKE + 4) == ALIGN             # bias must be 16-byte aligned
    assert fused(lib, Y=FAKE + 8) == ALIGN
    assert fused(lib, X=FAKE + 8) == ALIGN
    assert fused(lib, ws=None, wsb=0) == 11               # CCI_ERR_WORKSPACE
    assert fused(lib, wsb=64 * 64 * 2 - 2) == 11
    assert fused(lib, ws=FAKE + 8) == 11
    assert lib.cci_conv2d_fused(FAKE, 1, 1, 4, 4, 64, FAKE, FAKE, 64, 3, 3, 1, 1, 1, 1, 8, 2, None, 1, 1,
                                FAKE, None, None, 0, None) == 11
    assert lib.cci_conv2d_fused(FAKE, 1, 1, 4, 4, 64, FAKE, FAKE, 64, 3, 3, 1, 1, 1, 1, 8, 2, None, 1, 7,
                                FAKE, None, FAKE, 1 << 20, None) == DTYPE


def test_pack_stats_rejects(lib):
    s = lib.cci_pack_stats
    assert s(FAKE, 5, 16, 8, 8, 2, FAKE, None) == DTYPE
    assert s(None, 1, 16, 8, 8, 2, FAKE, None) == NULL
    assert s(FAKE, 1, 16, 8, 8, 2, None, None) == NULL
    assert s(FAKE, 1, 0, 8, 8, 2, FAKE, None) == SHAPE
    assert s(FAKE, 1, 12, 8, 8, 2, FAKE, None) == GROUP
    assert s(FAKE, 1, 16, 8, 8, 9, FAKE, None) == GROUP
    assert s(FAKE + 1, 1, 16, 8, 8, 2, FAKE, None) == ALIGN
    assert s(FAKE, 1, 16, 8, 8, 2, FAKE + 4, None) == ALIGN


def test_td_mask_rejects(lib):
    t = lib.cci_td_mask
    assert t(FAKE, 5, 16, 8, 8, 2, 0.5, FAKE, FAKE, None, None, None) == DTYPE
    assert t(None, 0, 16, 8, 8, 2, 0.5, FAKE, FAKE, None, None, None) == NULL
    assert t(FAKE, 0, 16, 8, 8, 2, 0.5, None, FAKE, None, None, None) == NULL
    assert t(FAKE, 0, 16, 8, 8, 2, 0.5, FAKE, None, None, None, None) == NULL
    assert t(FAKE, 0, 16, 0, 8, 2, 0.5, FAKE, FAKE, None, None, None) == SHAPE
    assert t(FAKE, 0, 12, 8, 8, 2, 0.5, FAKE, FAKE, None, None, None) == GROUP
    assert t(FAKE, 0, 16, 8, 8, 2, 1.5, FAKE, FAKE, None, None, None) == VALUE
    assert t(FAKE, 0, 16, 8, 8, 2, -0.1, FAKE, FAKE, None, None, None) == VALUE
    assert t(FAKE, 0, 16, 8, 8, 2, float("nan"), FAKE, FAKE, None, None, None) == VALUE
    assert t(FAKE + 2, 0, 16, 8, 8, 2, 0.5, FAKE, FAKE, None, None, None) == ALIGN


def test_bbs_rejects(lib):
    p, f = lib.cci_bbs_pack, lib.cci_bbs_linear
    assert p(FAKE, 5, 16, 64, 8, 2, FAKE, FAKE, None, None) == DTYPE
    assert p(None, 1, 16, 64, 8, 2, FAKE, FAKE, None, None) == NULL
    assert p(FAKE, 1, 16, 60, 8, 2, FAKE, FAKE, None, None) == GROUP   # R % G
    assert p(FAKE, 1, 16, 64, 8, 9, FAKE, FAKE, None, None) == GROUP
    assert p(FAKE, 1, 0, 64, 8, 2, FAKE, FAKE, None, None) == SHAPE
    assert p(FAKE + 1, 1, 16, 64, 8, 2, FAKE, FAKE, None, None) == ALIGN
    assert f(FAKE, 1, 16, 60, FAKE, FAKE, 16, 8, 2, FAKE, None, 0, None, 0, None) == GROUP
    assert f(FAKE, 1, 16, 64, FAKE, FAKE, 16, 64, 2, FAKE, None, 1, None, 0, None) == UNSUP  # gather: 32 % G
    assert f(FAKE, 1, 16, 64, FAKE, FAKE, 16, 8, 2, FAKE, None, 2, None, 0, None) == UNSUP  # no such family
    assert f(FAKE, 1, 16, 64, FAKE, FAKE, 16, 8, 2, FAKE, None, 5, None, 0, None) == 11     # workspace
    assert f(FAKE, 1, 0, 64, FAKE, FAKE, 16, 8, 2, None, None, 1, None, 0, None) == OK      # empty
