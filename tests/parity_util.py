"""Helpers for comparing the CUDA path with the oracle.

The tolerance is the one fixed for this method's outputs: for every output
element, |y - y_oracle| <= 1e-5 * S with S = sum |w||x| over the kept terms
(fp32 accumulation against an fp64 reference; bf16 inputs are compared on
their exact values).  Where S == 0 every term is zero and y must be exactly 0.
Packed indices must match exactly and packed values bit for bit.
"""
from __future__ import annotations

import numpy as np
import torch

import oracle

TOL = 1e-5


def f64(t: torch.Tensor) -> np.ndarray:
    """Exact float64 copy of a float32 / bfloat16 tensor."""
    return t.detach().to("cpu").to(torch.float64).numpy()


def assert_pack_equal(values_gpu, idx_gpu, values_o, idx_o):
    vi = idx_gpu.to("cpu").numpy()
    assert vi.shape == idx_o.shape
    bad = np.argwhere(vi != idx_o)
    assert bad.size == 0, f"{len(bad)} index mismatches, first at {bad[:5].tolist()}"
    vg = f64(values_gpu)
    same = vg.view(np.int64) == np.ascontiguousarray(values_o).view(np.int64)
    assert same.all(), f"{(~same).sum()} value mismatches (bitwise)"


def assert_within_tol(y_gpu: np.ndarray, y_o: np.ndarray, S: np.ndarray, what: str = ""):
    assert y_gpu.shape == y_o.shape, (y_gpu.shape, y_o.shape)
    assert np.isfinite(y_gpu).all(), f"{what}: non-finite outputs"
    err = np.abs(y_gpu - y_o)
    lim = TOL * S
    bad = err > lim
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outputs out of tolerance; first at "
                             f"{i.tolist()}: gpu={y_gpu[tuple(i)]!r} oracle={y_o[tuple(i)]!r} "
                             f"S={S[tuple(i)]!r} err/S={err[tuple(i)] / max(S[tuple(i)], 1e-300):.3e}")
    zero = S == 0
    assert (y_gpu[zero] == 0).all(), f"{what}: nonzero output where every term is zero"


def oracle_reference(W: torch.Tensor, G: int, K: int):
    """Oracle pack + decompress of the dense weights W[Cout][R] (any dtype)."""
    v, i = oracle.pack(f64(W), G, K)
    Wd, mask = oracle.decompress(v, i, W.shape[0], G)
    return v, i, Wd, mask


def sample_rows(N: int, k: int, seed: int = 0) -> np.ndarray:
    """First and last rows (tile edges and the ragged tail) plus random ones."""
    if N <= k:
        return np.arange(N, dtype=np.int64)
    rng = np.random.default_rng(seed)
    edge = min(64, k // 4)
    mid = rng.choice(np.arange(edge, N - edge), size=k - 2 * edge, replace=False)
    return np.unique(np.concatenate([np.arange(edge), np.sort(mid), np.arange(N - edge, N)]))


def assert_fused_within_tol(y_gpu: np.ndarray, y_ref: np.ndarray, S: np.ndarray, out_bf16: bool, what: str = ""):
    """Outputs of the fused epilogue against oracle.epilogue(): the product's bound
    1e-5 * S (S including |bias|; ReLU is 1-Lipschitz) plus, for bf16 outputs, the
    final rounding (half a bf16 unit in the last place <= 2^-8 * |y|)."""
    assert y_gpu.shape == y_ref.shape, (y_gpu.shape, y_ref.shape)
    assert np.isfinite(y_gpu).all(), f"{what}: non-finite outputs"
    lim = TOL * (1 + 2.0 ** -8) * S + (2.0 ** -8 * np.abs(y_ref) if out_bf16 else 0.0)
    err = np.abs(y_gpu - y_ref)
    bad = err > lim
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outputs out of tolerance; first at "
                             f"{i.tolist()}: gpu={y_gpu[tuple(i)]!r} ref={y_ref[tuple(i)]!r} S={S[tuple(i)]!r}")
