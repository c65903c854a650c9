"""Python binding of libcci.so: CCI-sparse layers (arXiv 1910.11971) on GB300.

Argument marshalling only.  Every step of the computation runs in the CUDA
kernels of ``libcci.so`` (built from ``csrc/`` by ``build.py``); PyTorch is used
for device memory and the current stream.  There is no CPU path: if the
library is missing or a call fails, an exception is raised.

    values, idx = pack(W, G, K)                         # Sec. 3.1 / 5.1
    Y = linear(X, values, idx, Cout, G, K)              # Alg. 2, Y[N][Cout] fp32
    Y = conv2d(X, values, idx, Cout, G, K, KH, KW, stride, pad)  # NHWC

Layouts are those of ``include/cci.h``: W [Cout][R], values/idx [Cout/G][R][K],
X [N][Cin] (product) or NHWC [B][H][W][Cin] (convolution), Y fp32.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libcci.so")

F32, BF16 = 0, 1
ALGO_AUTO, ALGO_GENERIC, ALGO_REGTILE, ALGO_DENSE_TC, ALGO_EXPAND, ALGO_DENSE_TC_WS = 0, 1, 2, 3, 4, 5

STATUS_NAMES = {
    0: "CCI_OK", 1: "CCI_ERR_NULL", 2: "CCI_ERR_SHAPE", 3: "CCI_ERR_GROUP", 4: "CCI_ERR_DTYPE",
    5: "CCI_ERR_ALIGN", 6: "CCI_ERR_VALUE", 7: "CCI_ERR_CUDA", 8: "CCI_ERR_TIMEOUT",
    9: "CCI_ERR_UNSUPPORTED", 10: "CCI_ERR_INDEX", 11: "CCI_ERR_WORKSPACE",
}

# exported symbols with their ctypes signatures (the declarations of cci.h)
_P, _I64, _I32, _U32P = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
SIGNATURES = {
    "cci_pack": (_I32, [_P, _I32, _I64, _I64, _I32, _I32, _P, _P, _U32P, _P]),
    "cci_linear": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _U32P, _P]),
    "cci_linear_ex": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _U32P, _I32, _P]),
    "cci_conv2d": (_I32, [_P, _I32, _I64, _I64, _I64, _I64, _P, _P, _I64, _I32, _I32, _I32, _I32,
                          _I32, _I32, _I32, _I32, _P, _U32P, _P]),
    "cci_conv2d_ex": (_I32, [_P, _I32, _I64, _I64, _I64, _I64, _P, _P, _I64, _I32, _I32, _I32, _I32,
                             _I32, _I32, _I32, _I32, _P, _U32P, _I32, _P]),
    "cci_linear_ws": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _U32P, _I32, _P,
                             ctypes.c_size_t, _P]),
    "cci_conv2d_ws": (_I32, [_P, _I32, _I64, _I64, _I64, _I64, _P, _P, _I64, _I32, _I32, _I32, _I32,
                             _I32, _I32, _I32, _I32, _P, _U32P, _I32, _P, ctypes.c_size_t, _P]),
    "cci_linear_fused": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _I32, _I32, _P,
                                _U32P, _P, ctypes.c_size_t, _P]),
    "cci_conv2d_fused": (_I32, [_P, _I32, _I64, _I64, _I64, _I64, _P, _P, _I64, _I32, _I32, _I32,
                                _I32, _I32, _I32, _I32, _I32, _P, _I32, _I32, _P, _U32P, _P,
                                ctypes.c_size_t, _P]),
    "cci_pack_stats": (_I32, [_P, _I32, _I64, _I64, _I32, _I32, _P, _P]),
    "cci_bbs_pack": (_I32, [_P, _I32, _I64, _I64, _I32, _I32, _P, _P, _U32P, _P]),
    "cci_bbs_linear": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _U32P, _I32, _P,
                              ctypes.c_size_t, _P]),
    "cci_td_mask": (_I32, [_P, _I32, _I64, _I64, _I32, _I32, ctypes.c_float, _P, _P, _P, _U32P, _P]),
    "cci_td_drop_rate": (ctypes.c_float, [_I64, _I64, ctypes.c_float, ctypes.c_float]),
    "cci_workspace_size": (ctypes.c_size_t, [_I32, _I32, _I64, _I64]),
    "cci_linear_host_buffer_size": (ctypes.c_size_t, [_I32, _I64, _I64, _I64]),
    "cci_linear_host": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _I64, _P,
                               ctypes.c_size_t, _U32P, _P, _P, _P]),
    "cci_linear_dense_tc_static": (_I32, [_P, _I32, _I64, _I64, _P, _P, _I64, _I32, _I32, _P, _U32P,
                                          _P]),
    "cci_dense_linear_tc": (_I32, [_P, _I32, _I64, _I64, _P, _I64, _P, _U32P, _P]),
    "cci_dense_planes": (_I32, [_P, _I32, _I64, _I64, _P, ctypes.c_size_t, _P]),
    "cci_dense_conv2d_tc": (_I32, [_P, _I32, _I64, _I64, _I64, _I64, _P, _I64, _I32, _I32, _I32, _I32,
                                   _I32, _I32, _P, _U32P, _P]),
    "cci_kernel_name": (ctypes.c_char_p, [_I32, _I64, _I64, _I64, _I32, _I32, _I32]),
    "cci_status_string": (ctypes.c_char_p, [_I32]),
    "cci_decode_device_status": (_I32, [ctypes.c_uint32]),
    "cci_version": (_I32, []),
    "cci_fma_probe": (_I32, [_P, _I32, _I32, _I32, _P]),
    "cci_wait_probe": (_I32, [_U32P, _I32, _P]),
}

_lib = None


class CCIError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = int(status)
        text = lib().cci_status_string(self.status).decode() if _lib is not None else ""
        super().__init__(f"{where}: {STATUS_NAMES.get(self.status, self.status)} ({text})")


def lib() -> ctypes.CDLL:
    """The loaded libcci.so.  Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"libcci.so is not built ({LIB_PATH}); run "
                               "`python -m paper_1910_11971_gb300.build` (needs nvcc)")
        h = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(h, name)
            fn.restype = res
            fn.argtypes = args
        _lib = h
    return _lib


def status_string(code: int) -> str:
    return lib().cci_status_string(int(code)).decode()


def decode_status(word: int) -> int:
    return int(lib().cci_decode_device_status(ctypes.c_uint32(int(word) & 0xffffffff)))


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.float32:
        return F32
    if t.dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported dtype {t.dtype}: float32 or bfloat16")


def _stream(device: torch.device) -> int:
    return torch.cuda.current_stream(device).cuda_stream


def _cuda_contig(t: torch.Tensor, name: str) -> None:
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _check(code: int, where: str) -> None:
    if code != 0:
        raise CCIError(code, where)


def new_status(device) -> torch.Tensor:
    """A zeroed device status word for the ``status=`` argument of the calls."""
    return torch.zeros(1, dtype=torch.int32, device=device)


def read_status(status: torch.Tensor) -> int:
    """Synchronise and return the first error recorded in a status word (0 = none)."""
    return decode_status(int(status.item()))


def pack(W: torch.Tensor, G: int, K: int, *, status: Optional[torch.Tensor] = None,
         check: bool = True, out: Optional[Tuple[torch.Tensor, torch.Tensor]] = None):
    """Per-group top-K by |w| (ties to the lower index) -> (values, idx).

    W: CUDA [Cout][R] float32 or bfloat16.  With ``check`` (the default) the call
    synchronises and raises on NaN weights; with ``check=False`` it stays
    asynchronous and records errors only in ``status`` (if given)."""
    _cuda_contig(W, "W")
    Cout, R = W.shape
    if G < 1 or Cout % G:
        raise CCIError(3, "pack")
    if out is None:
        values = torch.empty((Cout // G, R, K), dtype=W.dtype, device=W.device)
        idx = torch.empty((Cout // G, R, K), dtype=torch.uint8, device=W.device)
    else:
        values, idx = out
    own_status = status is None and check
    if own_status:
        status = new_status(W.device)
    code = lib().cci_pack(W.data_ptr(), _dtype_code(W), Cout, R, G, K, values.data_ptr(),
                          idx.data_ptr(), status.data_ptr() if status is not None else None,
                          _stream(W.device))
    _check(code, "cci_pack")
    if check:
        dev = read_status(status)
        if dev:
            raise CCIError(dev, "cci_pack (device)")
    return values, idx


def workspace_size(algo: int, dtype: torch.dtype, Cout: int, R: int) -> int:
    """Bytes of workspace the kernel family needs for a layer (0: none)."""
    return int(lib().cci_workspace_size(algo, F32 if dtype == torch.float32 else BF16, Cout, R))


def new_workspace(algo: int, dtype: torch.dtype, Cout: int, R: int, device) -> Optional[torch.Tensor]:
    n = workspace_size(algo, dtype, Cout, R)
    return torch.empty(n, dtype=torch.uint8, device=device) if n else None


def _ws(workspace: Optional[torch.Tensor]):
    if workspace is None:
        return None, 0
    return workspace.data_ptr(), workspace.numel() * workspace.element_size()


def linear(X: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int, *,
           out: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
           algo: int = ALGO_AUTO, workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y[N][Cout] (fp32) = the CCI-sparse product of X[N][Cin] (Alg. 2).

    ``workspace``: device buffer for the families that need one (see
    ``workspace_size``); with ``algo`` AUTO or ``ALGO_DENSE_TC_WS`` and none given,
    the one that family asks for is allocated here from PyTorch memory (the
    library allocates nothing), so AUTO can reach its fastest family."""
    _cuda_contig(X, "X")
    N, Cin = X.shape
    if workspace is None and algo == ALGO_AUTO:
        workspace = auto_workspace(X.dtype, Cin, Cin, Cout, G, K, X.device)
    elif workspace is None and algo == ALGO_DENSE_TC_WS:
        workspace = new_workspace(algo, X.dtype, Cout, Cin, X.device)
    Y = out if out is not None else torch.empty((N, Cout), dtype=torch.float32, device=X.device)
    wp, wb = _ws(workspace)
    code = lib().cci_linear_ws(X.data_ptr(), _dtype_code(X), N, Cin, values.data_ptr(),
                               idx.data_ptr(), Cout, G, K, Y.data_ptr(),
                               status.data_ptr() if status is not None else None, algo, wp, wb,
                               _stream(X.device))
    _check(code, "cci_linear")
    return Y


_copy_streams = {}


def host_chunk(N: int) -> int:
    """Default columns per chunk of ``linear_host``: about an eighth of N, in
    whole 128-column tiles."""
    eighth = (N + 7) // 8
    return max(128, (eighth + 127) // 128 * 128)


def host_buffer(dtype: torch.dtype, Cin: int, Cout: int, chunk: int, device) -> torch.Tensor:
    """A device buffer for ``linear_host`` (the library allocates nothing)."""
    n = lib().cci_linear_host_buffer_size(F32 if dtype == torch.float32 else BF16, Cin, Cout, chunk)
    if not n:
        raise ValueError("cci_linear_host_buffer_size: invalid shape")
    return torch.empty(n, dtype=torch.uint8, device=device)


def linear_host(X_host: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int, *,
                out: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                chunk: Optional[int] = None, buffer: Optional[torch.Tensor] = None) -> torch.Tensor:
    """``linear`` with X and Y in host memory (``cci_linear_host``): column chunks
    are copied in, multiplied and copied out on three streams, overlapping.
    X_host should be pinned; the result ``out`` (pinned fp32 [N][Cout], allocated
    when not given) is complete once the device's current stream has been
    synchronised."""
    if X_host.is_cuda or not X_host.is_contiguous():
        raise ValueError("X_host must be a contiguous host tensor")
    dev = values.device
    N, Cin = X_host.shape
    chunk = chunk or host_chunk(N)
    if buffer is None:
        buffer = host_buffer(X_host.dtype, Cin, Cout, chunk, dev)
    Y = out if out is not None else torch.empty((N, Cout), dtype=torch.float32).pin_memory()
    if Y.is_cuda or not Y.is_contiguous() or Y.dtype != torch.float32:
        raise ValueError("out must be a contiguous fp32 host tensor")
    key = (dev.index if dev.index is not None else torch.cuda.current_device())
    if key not in _copy_streams:
        _copy_streams[key] = (torch.cuda.Stream(dev), torch.cuda.Stream(dev))
    s_in, s_out = _copy_streams[key]
    code = lib().cci_linear_host(X_host.data_ptr(), _dtype_code(X_host), N, Cin, values.data_ptr(),
                                 idx.data_ptr(), Cout, G, K, Y.data_ptr(), chunk, buffer.data_ptr(),
                                 buffer.numel(), status.data_ptr() if status is not None else None,
                                 _stream(dev), s_in.cuda_stream, s_out.cuda_stream)
    _check(code, "cci_linear_host")
    return Y


def conv_out_hw(H: int, W: int, KH: int, KW: int, stride: Sequence[int], pad: Sequence[int]):
    return (H + 2 * pad[0] - KH) // stride[0] + 1, (W + 2 * pad[1] - KW) // stride[1] + 1


def conv2d(X: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int,
           KH: int, KW: int, stride=(1, 1), pad=(0, 0), *, out: Optional[torch.Tensor] = None,
           status: Optional[torch.Tensor] = None, algo: int = ALGO_AUTO,
           workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y NHWC [B][P][Q][Cout] (fp32) = CCI-sparse convolution of X NHWC [B][H][W][Cin]."""
    _cuda_contig(X, "X")
    B, H, W, Cin = X.shape
    P, Q = conv_out_hw(H, W, KH, KW, stride, pad)
    Y = out if out is not None else torch.empty((B, max(P, 0), max(Q, 0), Cout), dtype=torch.float32,
                                                device=X.device)
    if workspace is None and algo == ALGO_AUTO:
        workspace = auto_workspace(X.dtype, Cin, KH * KW * Cin, Cout, G, K, X.device, max(stride))
    elif workspace is None and algo == ALGO_DENSE_TC_WS:
        workspace = new_workspace(algo, X.dtype, Cout, KH * KW * Cin, X.device)
    wp, wb = _ws(workspace)
    code = lib().cci_conv2d_ws(X.data_ptr(), _dtype_code(X), B, H, W, Cin, values.data_ptr(),
                               idx.data_ptr(), Cout, KH, KW, stride[0], stride[1], pad[0], pad[1],
                               G, K, Y.data_ptr(), status.data_ptr() if status is not None else None,
                               algo, wp, wb, _stream(X.device))
    _check(code, "cci_conv2d")
    return Y


def bbs_pack(W: torch.Tensor, G: int, K: int, *, status: Optional[torch.Tensor] = None):
    """(values[Cout][R/G][K], idx[Cout][R/G][K]) of the balanced-sparse form of W
    (groups of G consecutive inputs; ``cci_bbs_pack``)."""
    _cuda_contig(W, "W")
    Cout, R = W.shape
    values = torch.empty((Cout, R // G, K), dtype=W.dtype, device=W.device)
    idx = torch.empty((Cout, R // G, K), dtype=torch.uint8, device=W.device)
    _check(lib().cci_bbs_pack(W.data_ptr(), _dtype_code(W), Cout, R, G, K, values.data_ptr(), idx.data_ptr(),
                              status.data_ptr() if status is not None else None, _stream(W.device)),
           "cci_bbs_pack")
    return values, idx


def bbs_linear(X: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int, *,
               out: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
               algo: int = ALGO_AUTO, workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y[N][Cout] (fp32) = the balanced-sparse product (``cci_bbs_linear``); with AUTO
    or ALGO_DENSE_TC_WS and no workspace, one is allocated here."""
    _cuda_contig(X, "X")
    N, Cin = X.shape
    if workspace is None and algo in (ALGO_AUTO, ALGO_DENSE_TC_WS):
        workspace = new_workspace(ALGO_DENSE_TC_WS, X.dtype, Cout, Cin, X.device)
    Y = out if out is not None else torch.empty((N, Cout), dtype=torch.float32, device=X.device)
    wp, wb = _ws(workspace)
    _check(lib().cci_bbs_linear(X.data_ptr(), _dtype_code(X), N, Cin, values.data_ptr(), idx.data_ptr(), Cout,
                                G, K, Y.data_ptr(), status.data_ptr() if status is not None else None, algo, wp,
                                wb, _stream(X.device)), "cci_bbs_linear")
    return Y


def td_mask(W: torch.Tensor, G: int, K: int, rate: float, uniforms: torch.Tensor, *,
            out: Optional[torch.Tensor] = None, mask: Optional[torch.Tensor] = None,
            status: Optional[torch.Tensor] = None):
    """(W_out, mask) of one targeted-dropout step (``cci_td_mask``): candidates (the
    weights packing would drop) zeroed where ``uniforms < rate``."""
    _cuda_contig(W, "W")
    _cuda_contig(uniforms, "uniforms")
    Cout, R = W.shape
    Wo = out if out is not None else torch.empty_like(W)
    m = mask if mask is not None else torch.empty((Cout, R), dtype=torch.uint8, device=W.device)
    _check(lib().cci_td_mask(W.data_ptr(), _dtype_code(W), Cout, R, G, K, float(rate), uniforms.data_ptr(),
                             Wo.data_ptr(), m.data_ptr(), status.data_ptr() if status is not None else None,
                             _stream(W.device)), "cci_td_mask")
    return Wo, m


def td_drop_rate(step: int, ramp_steps: int, start: float = 0.5, end: float = 1.0) -> float:
    """The candidate drop rate of Sec. 5.1 at ``step`` (``cci_td_drop_rate``): from
    ``start`` (50 %) toward ``end`` (100 %), linear over ``ramp_steps`` steps and then
    constant (the paper fixes the end points only)."""
    return float(lib().cci_td_drop_rate(int(step), int(ramp_steps), float(start), float(end)))


def pack_stats(W: torch.Tensor, G: int, K: int, counts: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Adds (nonzero weights of W, nonzero weights packing with (G, K) drops) into
    ``counts`` (int64 device tensor of 2, zeroed here when not given) and returns it
    (``cci_pack_stats``; read it after a sync)."""
    _cuda_contig(W, "W")
    Cout, R = W.shape
    if counts is None:
        counts = torch.zeros(2, dtype=torch.int64, device=W.device)
    _check(lib().cci_pack_stats(W.data_ptr(), _dtype_code(W), Cout, R, G, K, counts.data_ptr(),
                                _stream(W.device)), "cci_pack_stats")
    return counts


def _out_code(dtype: torch.dtype) -> int:
    if dtype == torch.float32:
        return F32
    if dtype == torch.bfloat16:
        return BF16
    raise TypeError(f"unsupported output dtype {dtype}: float32 or bfloat16")


def linear_fused(X: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int, *,
                 bias: Optional[torch.Tensor] = None, relu: bool = False,
                 out_dtype: torch.dtype = torch.float32, out: Optional[torch.Tensor] = None,
                 status: Optional[torch.Tensor] = None,
                 workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y[N][Cout] = relu?(product + bias) in ``out_dtype`` (fp32 or bf16), on a
    tensor-core family (``cci_linear_fused``: the fused one where AUTO takes it,
    else the workspace one, whose workspace is allocated here when not given)."""
    _cuda_contig(X, "X")
    N, Cin = X.shape
    if workspace is None and not kernel_name(X.dtype, Cin, Cin, Cout, G, K).startswith("dense_tc_fused"):
        workspace = new_workspace(ALGO_DENSE_TC_WS, X.dtype, Cout, Cin, X.device)
    Y = out if out is not None else torch.empty((N, Cout), dtype=out_dtype, device=X.device)
    if bias is not None:
        _cuda_contig(bias, "bias")
    wp, wb = _ws(workspace)
    code = lib().cci_linear_fused(X.data_ptr(), _dtype_code(X), N, Cin, values.data_ptr(), idx.data_ptr(),
                                  Cout, G, K, bias.data_ptr() if bias is not None else None, int(relu),
                                  _out_code(Y.dtype), Y.data_ptr(),
                                  status.data_ptr() if status is not None else None, wp, wb,
                                  _stream(X.device))
    _check(code, "cci_linear_fused")
    return Y


def conv2d_fused(X: torch.Tensor, values: torch.Tensor, idx: torch.Tensor, Cout: int, G: int, K: int,
                 KH: int, KW: int, stride=(1, 1), pad=(0, 0), *, bias: Optional[torch.Tensor] = None,
                 relu: bool = False, out_dtype: torch.dtype = torch.float32,
                 out: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None,
                 workspace: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y NHWC [B][P][Q][Cout] = relu?(convolution + bias) in ``out_dtype`` (fp32 or
    bf16), on a tensor-core family (``cci_conv2d_fused``, as ``linear_fused``)."""
    _cuda_contig(X, "X")
    B, H, W, Cin = X.shape
    P, Q = conv_out_hw(H, W, KH, KW, stride, pad)
    Y = out if out is not None else torch.empty((B, max(P, 0), max(Q, 0), Cout), dtype=out_dtype,
                                                device=X.device)
    fused = kernel_name(X.dtype, Cin, KH * KW * Cin, Cout, G, K).startswith("dense_tc_fused") and max(stride) <= 2
    if workspace is None and not fused:
        workspace = new_workspace(ALGO_DENSE_TC_WS, X.dtype, Cout, KH * KW * Cin, X.device)
    if bias is not None:
        _cuda_contig(bias, "bias")
    wp, wb = _ws(workspace)
    code = lib().cci_conv2d_fused(X.data_ptr(), _dtype_code(X), B, H, W, Cin, values.data_ptr(),
                                  idx.data_ptr(), Cout, KH, KW, stride[0], stride[1], pad[0], pad[1], G, K,
                                  bias.data_ptr() if bias is not None else None, int(relu),
                                  _out_code(Y.dtype), Y.data_ptr(),
                                  status.data_ptr() if status is not None else None, wp, wb,
                                  _stream(X.device))
    _check(code, "cci_conv2d_fused")
    return Y


def dense_planes(W: torch.Tensor) -> torch.Tensor:
    """Dense weights W[Cout][R] (OHWI rows for a convolution) in the workspace
    layout of the dense tensor-core family (``cci_dense_planes``), for
    ``dense_linear_tc`` / ``dense_conv2d_tc``: bf16 as is, fp32 as its two
    operand planes (a byte tensor)."""
    _cuda_contig(W, "W")
    Cout = W.shape[0]
    R = W.numel() // Cout
    Wd = new_workspace(ALGO_DENSE_TC_WS, W.dtype, Cout, R, W.device)
    _check(lib().cci_dense_planes(W.data_ptr(), _dtype_code(W), Cout, R, Wd.data_ptr(), Wd.numel(),
                                  _stream(W.device)), "cci_dense_planes")
    return Wd


def dense_linear_tc(X: torch.Tensor, Wd: torch.Tensor, Cout: int, *, out: Optional[torch.Tensor] = None,
                    status: Optional[torch.Tensor] = None) -> torch.Tensor:
    """Y[N][Cout] = X Wd^T on the library's tensor-core GEMM with dense weights and
    no decompression (``cci_dense_linear_tc``).  Wd is the dense family's workspace
    layout, as ``dense_planes`` writes it."""
    _cuda_contig(X, "X")
    _cuda_contig(Wd, "Wd")
    N, Cin = X.shape
    Y = out if out is not None else torch.empty((N, Cout), dtype=torch.float32, device=X.device)
    _check(lib().cci_dense_linear_tc(X.data_ptr(), _dtype_code(X), N, Cin, Wd.data_ptr(), Cout, Y.data_ptr(),
                                     status.data_ptr() if status is not None else None, _stream(X.device)),
           "cci_dense_linear_tc")
    return Y


def dense_conv2d_tc(X: torch.Tensor, Wd: torch.Tensor, Cout: int, KH: int, KW: int, stride=(1, 1), pad=(0, 0), *,
                    out: Optional[torch.Tensor] = None, status: Optional[torch.Tensor] = None) -> torch.Tensor:
    """NHWC convolution on the library's tensor-core GEMM with dense OHWI weights in
    the dense family's workspace layout and no decompression (``cci_dense_conv2d_tc``)."""
    _cuda_contig(X, "X")
    _cuda_contig(Wd, "Wd")
    B, H, W, Cin = X.shape
    P, Q = conv_out_hw(H, W, KH, KW, stride, pad)
    Y = out if out is not None else torch.empty((B, max(P, 0), max(Q, 0), Cout), dtype=torch.float32,
                                                device=X.device)
    _check(lib().cci_dense_conv2d_tc(X.data_ptr(), _dtype_code(X), B, H, W, Cin, Wd.data_ptr(), Cout, KH, KW,
                                     stride[0], stride[1], pad[0], pad[1], Y.data_ptr(),
                                     status.data_ptr() if status is not None else None, _stream(X.device)),
           "cci_dense_conv2d_tc")
    return Y


def kernel_name(dtype: torch.dtype, Cin: int, R: int, Cout: int, G: int, K: int,
                algo: int = ALGO_AUTO) -> str:
    """The kernel family a call would run (``cci_kernel_name``; for AUTO: given the
    workspace ``auto_workspace`` provides)."""
    code = F32 if dtype == torch.float32 else BF16
    return lib().cci_kernel_name(code, Cin, R, Cout, G, K, algo).decode()


def auto_workspace(dtype: torch.dtype, Cin: int, R: int, Cout: int, G: int, K: int,
                   device, stride: int = 1) -> Optional[torch.Tensor]:
    """The workspace AUTO needs to reach its fastest family for a layer (R = Cin
    for a product, KH*KW*Cin for a convolution of the given largest stride), from
    PyTorch memory: None when that family needs none (the library allocates
    nothing itself)."""
    name = kernel_name(dtype, Cin, R, Cout, G, K, ALGO_AUTO)
    if name.startswith("dense_tc_fused") and stride <= 2:
        return None
    if not lib().cci_kernel_name(F32 if dtype == torch.float32 else BF16, Cin, R, Cout, G, K, ALGO_DENSE_TC_WS):
        return None
    return new_workspace(ALGO_DENSE_TC_WS, dtype, Cout, R, device)


def fma_probe(out: torch.Tensor, blocks: int, threads: int, iters: int) -> None:
    _check(lib().cci_fma_probe(out.data_ptr(), blocks, threads, iters, _stream(out.device)),
           "cci_fma_probe")
