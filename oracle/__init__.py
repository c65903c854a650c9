"""fp64 CPU oracle for CCI-sparse layers (arXiv 1910.11971).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg may import this package.  The CUDA library never
calls it, and it shares no code with the CUDA library: the arithmetic lives in
``cci_oracle.c`` (plain C, fp64); this module only marshals numpy arrays.

Routines (inputs are float64 arrays holding the exact values of the storage
dtype; outputs are float64):

* ``pack(W, G, K)``  -- Sec. 5.1 magnitude selection under the group constraint
  of Sec. 3.1: per (group, r) keep the K largest |w|, ties to the lower index,
  emitted in increasing index.
* ``decompress(values, idx, Cout, G)`` -- back to the dense M x N matrix W-hat of
  Sec. 3.1, with a count of the slots landing on each entry.
* ``linear(X, Wd, mask)`` -- Alg. 1 on the decompressed matrix, plus the error
  scale S = sum |w||x| over the same terms.
* ``linear_alg2(X, values, idx, Cout, G)`` -- Alg. 2 taken literally.
* ``conv2d(X, Wd, mask, ...)`` -- direct convolution (NHWC input, OHWI weights).
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import math
from fractions import Fraction

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
SOURCE = os.path.join(_HERE, "cci_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB = os.path.join(_BUILD, "liboracle.so")


def build(force: bool = False, src: str = SOURCE, out: str = _LIB) -> str:
    """Compile ``cci_oracle.c`` (or a copy of it at ``src``) into a shared library."""
    if not force and os.path.exists(out) and os.path.getmtime(out) >= os.path.getmtime(src):
        return out
    os.makedirs(os.path.dirname(out), exist_ok=True)
    tmp = out + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", src, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True, capture_output=True)
    except subprocess.CalledProcessError:
        # no OpenMP runtime: the same code on one thread
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, out)
    return out


class OracleError(RuntimeError):
    def __init__(self, code: int, what: str):
        super().__init__(f"oracle {what} returned status {code}")
        self.code = code


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a: np.ndarray):
    return a.ctypes.data_as(ctypes.c_void_p)


def conv_out_hw(H: int, W: int, KH: int, KW: int, sh: int, sw: int, ph: int, pw: int):
    return (H + 2 * ph - KH) // sh + 1, (W + 2 * pw - KW) // sw + 1


class Oracle:
    """One loaded build of ``cci_oracle.c``."""

    def __init__(self, libpath: str):
        lib = ctypes.CDLL(libpath)
        p, i64, i32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int
        lib.oracle_threads.restype = i32
        lib.oracle_pack.argtypes = [p, i64, i64, i32, i32, p, p]
        lib.oracle_pack.restype = i32
        lib.oracle_decompress.argtypes = [p, p, i64, i64, i32, i32, p, p]
        lib.oracle_decompress.restype = i32
        lib.oracle_linear.argtypes = [p, i64, i64, p, p, i64, p, p]
        lib.oracle_linear.restype = None
        lib.oracle_linear_alg2.argtypes = [p, i64, i64, p, p, i64, i32, i32, p]
        lib.oracle_linear_alg2.restype = i32
        lib.oracle_conv2d.argtypes = [p, i64, i64, i64, i64, p, p, i64, i32, i32, i32, i32,
                                      i32, i32, p, i64, p, p]
        lib.oracle_conv2d.restype = i32
        self.lib = lib
        self.path = libpath

    def threads(self) -> int:
        return int(self.lib.oracle_threads())

    def pack(self, W, G: int, K: int):
        """W[Cout][R] -> (values[Cout/G][R][K] float64, idx[Cout/G][R][K] uint8)."""
        W = _f64(W)
        Cout, R = W.shape
        ng = Cout // G if G > 0 and Cout % G == 0 else 0
        values = np.zeros((max(ng, 1), R, max(K, 1)), np.float64)
        idx = np.zeros((max(ng, 1), R, max(K, 1)), np.uint8)
        st = self.lib.oracle_pack(_ptr(W), Cout, R, G, K, _ptr(values), _ptr(idx))
        if st:
            raise OracleError(st, "pack")
        return values, idx

    def decompress(self, values, idx, Cout: int, G: int):
        """(values, idx) -> (Wd[Cout][R] float64, mask[Cout][R] int32 slot counts)."""
        values = _f64(values)
        idx = np.ascontiguousarray(idx, dtype=np.uint8)
        _, R, K = values.shape
        Wd = np.zeros((Cout, R), np.float64)
        mask = np.zeros((Cout, R), np.int32)
        st = self.lib.oracle_decompress(_ptr(values), _ptr(idx), Cout, R, G, K, _ptr(Wd),
                                        _ptr(mask))
        if st:
            raise OracleError(st, "decompress")
        return Wd, mask

    def linear(self, X, Wd, mask):
        """Y[N][Cout] = X @ Wd^T over the kept entries, and S = |X| @ |Wd|^T likewise."""
        X = _f64(X)
        Wd = _f64(Wd)
        mask = np.ascontiguousarray(mask, dtype=np.int32)
        N, R = X.shape
        Cout = Wd.shape[0]
        Y = np.empty((N, Cout), np.float64)
        S = np.empty((N, Cout), np.float64)
        self.lib.oracle_linear(_ptr(X), N, R, _ptr(Wd), _ptr(mask), Cout, _ptr(Y), _ptr(S))
        return Y, S

    def linear_alg2(self, X, values, idx, Cout: int, G: int):
        X = _f64(X)
        values = _f64(values)
        idx = np.ascontiguousarray(idx, dtype=np.uint8)
        N, R = X.shape
        K = values.shape[2]
        Y = np.empty((N, Cout), np.float64)
        st = self.lib.oracle_linear_alg2(_ptr(X), N, R, _ptr(values), _ptr(idx), Cout, G, K,
                                         _ptr(Y))
        if st:
            raise OracleError(st, "linear_alg2")
        return Y

    def conv2d(self, X, Wd, mask, KH: int, KW: int, stride=(1, 1), pad=(0, 0), pts=None):
        """X NHWC [B][H][W][Cin], Wd [Cout][KH*KW*Cin] (OHWI) -> (Y, S) at the output
        positions ``pts`` (flattened (b*P + p)*Q + q), or at all of them ([B*P*Q][Cout])."""
        X = _f64(X)
        Wd = _f64(Wd)
        mask = np.ascontiguousarray(mask, dtype=np.int32)
        B, H, Wi, Cin = X.shape
        Cout = Wd.shape[0]
        P, Q = conv_out_hw(H, Wi, KH, KW, stride[0], stride[1], pad[0], pad[1])
        if pts is None:
            npts, pts_arr = B * P * Q, None
        else:
            pts_arr = np.ascontiguousarray(pts, dtype=np.int64)
            npts = pts_arr.shape[0]
        Y = np.empty((npts, Cout), np.float64)
        S = np.empty((npts, Cout), np.float64)
        st = self.lib.oracle_conv2d(_ptr(X), B, H, Wi, Cin, _ptr(Wd), _ptr(mask), Cout, KH, KW,
                                    stride[0], stride[1], pad[0], pad[1],
                                    None if pts_arr is None else _ptr(pts_arr), npts, _ptr(Y),
                                    _ptr(S))
        if st:
            raise OracleError(st, "conv2d")
        return Y, S


_default = None


def allocation_error(G: int, Ps: float) -> float:
    """Eq. 1 (Sec. 4): probability that a nonzero weight finds no encoding slot
    when each of the G weights of a group is nonzero independently with
    probability 1 - Ps and the group has s = G * (1 - Ps) slots:
    sum over i > s of (i - s) * Binomial(i; G, 1 - Ps), divided by s."""
    s = G * (1.0 - Ps)
    si = int(round(s))
    if si < 1 or abs(s - si) > 1e-9:
        raise ValueError("s = G * (1 - Ps) must be a positive integer")
    p = 1.0 - Ps
    total = 0.0
    for i in range(si + 1, G + 1):
        total += (i - si) * math.comb(G, i) * p ** i * (1.0 - p) ** (G - i)
    return total / si


def allocation_error_exact(G: int, Ps) -> Fraction:
    """Eq. 1 in exact rational arithmetic (Ps a Fraction or a string such as '3/4')."""
    Ps = Fraction(Ps)
    p = 1 - Ps
    s = G * p
    if s.denominator != 1 or s < 1:
        raise ValueError("s = G * (1 - Ps) must be a positive integer")
    si = int(s)
    total = Fraction(0)
    for i in range(si + 1, G + 1):
        total += (i - si) * math.comb(G, i) * p ** i * (1 - p) ** (G - i)
    return total / si


def bbs_pack(W, G: int, K: int):
    """Balanced sparsity (Sec. 3.4, the comparison format): per output channel co
    and group of G consecutive inputs r in [g*G, g*G + G), the K weights of largest
    |w| (ties to the lower index) in increasing index; values[Cout][R/G][K] and
    idx[Cout][R/G][K] (offsets inside the group).  The same selection as CCI's
    pack on the transposed matrix, whose groups of G rows are G inputs."""
    W = _f64(W)
    Cout, R = W.shape
    if R % G:
        raise OracleError(2, "bbs_pack")
    v, i = pack(np.ascontiguousarray(W.T), G, K)  # [R/G][Cout][K]
    return np.ascontiguousarray(v.transpose(1, 0, 2)), np.ascontiguousarray(i.transpose(1, 0, 2))


def bbs_decompress(values, idx, R: int):
    """Dense Wd[Cout][R] and mask of a balanced-sparse matrix (repeated indices add)."""
    values = _f64(values)
    idx = np.asarray(idx)
    Cout, ng, K = values.shape
    G = R // ng
    Wd = np.zeros((Cout, R))
    mask = np.zeros((Cout, R), dtype=np.int32)
    for g in range(ng):
        for s in range(K):
            j = idx[:, g, s].astype(np.int64)
            if (j >= G).any():
                raise OracleError(6, "bbs_decompress")
            np.add.at(Wd, (np.arange(Cout), g * G + j), values[:, g, s])
            np.add.at(mask, (np.arange(Cout), g * G + j), 1)
    return Wd, mask


def td_mask(W, G: int, K: int, rate: float, u):
    """Targeted dropout for CCI training (Sec. 5.1): the weights that packing keeps
    are protected; each other weight (a pruning candidate) is dropped when its
    uniform draw is below the rate (both compared as fp32).  Returns (W_out, mask)."""
    W = _f64(W)
    Cout, R = W.shape
    _, idx = pack(W, G, K)
    keep = np.zeros((Cout, R), dtype=bool)
    for gi in range(Cout // G):
        for s in range(K):
            keep[gi * G + idx[gi, :, s].astype(np.int64), np.arange(R)] = True
    drop = ~keep & (np.asarray(u, dtype=np.float32) < np.float32(rate))
    return np.where(drop, 0.0, W), (~drop).astype(np.uint8)


def pack_stats(W, G: int, K: int):
    """(nonzero weights of W[Cout][R], nonzero weights that packing with group size G
    and K slots cannot keep): per group (G consecutive output channels at one r,
    Sec. 3.1) the nonzeros beyond K, summed.  Plain counting."""
    W = np.asarray(W)
    Cout, R = W.shape
    if Cout % G:
        raise ValueError("Cout % G != 0")
    nz = (W.reshape(Cout // G, G, R) != 0).sum(axis=1)
    return int(nz.sum()), int(np.maximum(nz - K, 0).sum())


def epilogue(Y, S, bias=None, relu: bool = False):
    """The output stage of a CNN layer applied to the exact product (fp64): Y + bias
    per output channel (last axis), then max(., 0); with the error scale of the
    sum extended by |bias|.  (Not part of the paper's method; the network around
    a layer.)"""
    Y = np.array(Y, dtype=np.float64, copy=True)
    S = np.array(S, dtype=np.float64, copy=True)
    if bias is not None:
        b = _f64(bias).reshape(-1)
        Y += b
        S += np.abs(b)
    if relu:
        Y = np.maximum(Y, 0.0)
    return Y, S


def get() -> Oracle:
    """The oracle built from ``cci_oracle.c`` (compiled on first use)."""
    global _default
    if _default is None:
        _default = Oracle(build())
    return _default


def threads() -> int:
    return get().threads()


def pack(W, G: int, K: int):
    return get().pack(W, G, K)


def decompress(values, idx, Cout: int, G: int):
    return get().decompress(values, idx, Cout, G)


def linear(X, Wd, mask):
    return get().linear(X, Wd, mask)


def linear_alg2(X, values, idx, Cout: int, G: int):
    return get().linear_alg2(X, values, idx, Cout, G)


def conv2d(X, Wd, mask, KH: int, KW: int, stride=(1, 1), pad=(0, 0), pts=None):
    return get().conv2d(X, Wd, mask, KH, KW, stride, pad, pts)
