"""Python face of the fp64 CPU oracle (cola_oracle.c).  TEST INFRASTRUCTURE ONLY.

Definitions followed (arXiv 2502.10940):
  * forward  -- Sec. 3.2, Eq. (main-fwd): h = B sigma(A x); token-major
    Z = X A^T, H = sigma(Z), Y = H B^T.
  * backward -- Sec. 3.4, the "2x rule" (grad_x = W^T grad_h,
    grad_W = grad_h x^T) applied to both products with the chain rule
    through sigma: dZ = (dY B) * sigma'(Z), dB = dY^T H, dA = dZ^T X,
    dX = dZ A.
  * CoLA-M   -- Sec. 4.2 / App. C: only the rank-r activation is saved; H is
    recomputed from it in the backward.
  * fused q/k/v -- Fig. 4: the q, k and v auto-encoders read the same x, so
    they are three independent layers sharing X, and dX is their sum.
  * CoLA-M block recompute -- Sec. 4.2 / App. C: the up-projection B sigma(.)
    is recomputed in the backward from the saved Z: Y = sigma(Z) B^T.
  * gated MLP -- Fig. 4, Sec. 3.2, App. E: the gate and up layers read one
    x and their outputs are multiplied element-wise, M = Y_gate * Y_up (the
    input of the down layer); backward dY_gate = dM * Y_up, dY_up = dM * Y_gate.

Every function takes / returns numpy arrays.  Full routines take float64;
the *_bf16 routines take bf16 bit patterns (uint16) and widen them exactly.
"""
import ctypes
import os

import numpy as np

from .build import build as _build

__all__ = [
    "SIGMA", "MODE", "lib", "sigma", "dsigma", "round_bf16", "widen_bf16",
    "fwd", "bwd", "fwd_qkv", "bwd_qkv", "recompute_up", "rows_bf16", "dA_entries_bf16",
    "dB_entries_bf16", "num_threads", "gate_up_product", "gate_up_backward", "gated_fwd",
]

SIGMA = {"identity": 0, "silu": 1, "gelu": 2}
MODE = {"cola": 0, "cola_m": 1}

_lib = None
_D = ctypes.POINTER(ctypes.c_double)
_U16 = ctypes.POINTER(ctypes.c_uint16)
_L = ctypes.POINTER(ctypes.c_long)
_long = ctypes.c_long
_int = ctypes.c_int


def lib():
    global _lib
    if _lib is None:
        path = _build()
        l = ctypes.CDLL(path)
        l.oracle_sigma.restype = ctypes.c_double
        l.oracle_sigma.argtypes = [_int, ctypes.c_double]
        l.oracle_dsigma.restype = ctypes.c_double
        l.oracle_dsigma.argtypes = [_int, ctypes.c_double]
        l.oracle_round_bf16.restype = ctypes.c_double
        l.oracle_round_bf16.argtypes = [ctypes.c_double]
        for name in ("oracle_sigma_vec", "oracle_dsigma_vec"):
            getattr(l, name).argtypes = [_int, _D, _D, _long]
        l.oracle_round_bf16_vec.argtypes = [_D, _D, _long]
        l.oracle_fwd.argtypes = [_long, _long, _long, _long, _int, _int, _D, _D, _D, _D, _D, _D]
        l.oracle_bwd.argtypes = [_long, _long, _long, _long, _int, _int, _int,
                                 _D, _D, _D, _D, _D, _D, _D, _D, _D, _D]
        l.oracle_rows_bf16.argtypes = [_long, _long, _long, _int, _int, _U16, _long, _U16, _U16,
                                       _U16, _long, _long, _L, _D, _D, _D, _D, _D]
        l.oracle_dA_entries_bf16.argtypes = [_long, _long, _long, _long, _int, _int, _U16, _long,
                                             _U16, _U16, _U16, _long, _long, _L, _L, _D]
        l.oracle_dB_entries_bf16.argtypes = [_long, _long, _long, _int, _int, _U16, _long, _U16,
                                             _U16, _long, _long, _L, _L, _D]
        l.oracle_recompute_up.argtypes = [_long, _long, _long, _int, _D, _D, _D]
        l.oracle_gate_up_product.argtypes = [_long, _D, _D, _D]
        l.oracle_gate_up_backward.argtypes = [_long, _D, _D, _D, _D, _D]
        l.oracle_num_threads.restype = _int
        _lib = l
    return _lib


def num_threads() -> int:
    return int(lib().oracle_num_threads())


def _f64(a):
    a = np.ascontiguousarray(a, dtype=np.float64)
    return a, a.ctypes.data_as(_D)


def _out(shape):
    a = np.empty(shape, dtype=np.float64)
    return a, a.ctypes.data_as(_D)


def _u16(a):
    a = np.ascontiguousarray(a, dtype=np.uint16)
    return a, a.ctypes.data_as(_U16)


def _idx(a):
    a = np.ascontiguousarray(a, dtype=np.int64)
    return a, a.ctypes.data_as(_L)


def _sig(kind):
    return SIGMA[kind] if isinstance(kind, str) else int(kind)


def sigma(kind, z):
    z, pz = _f64(z)
    out, po = _out(z.shape)
    lib().oracle_sigma_vec(_sig(kind), pz, po, z.size)
    return out


def dsigma(kind, z):
    z, pz = _f64(z)
    out, po = _out(z.shape)
    lib().oracle_dsigma_vec(_sig(kind), pz, po, z.size)
    return out


def round_bf16(x):
    x, px = _f64(x)
    out, po = _out(x.shape)
    lib().oracle_round_bf16_vec(px, po, x.size)
    return out


def widen_bf16(bits):
    """bf16 bit patterns (uint16) -> float64, exactly."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def fwd(X, A, B, sigma="silu", round_store=False):
    """Eq. (main-fwd), token-major.  Returns (Z, H, Y)."""
    X, px = _f64(X)
    A, pa = _f64(A)
    B, pb = _f64(B)
    n, d_in = X.shape
    r = A.shape[0]
    d_out = B.shape[0]
    assert A.shape == (r, d_in) and B.shape == (d_out, r)
    Z, pz = _out((n, r))
    H, ph = _out((n, r))
    Y, py = _out((n, d_out))
    lib().oracle_fwd(n, d_in, d_out, r, _sig(sigma), int(bool(round_store)), px, pa, pb, pz, ph, py)
    return Z, H, Y


def bwd(X, A, B, dY, Z, H=None, sigma="silu", mode="cola", round_store=False):
    """Sec. 3.4 backward.  H is the saved H (CoLA); CoLA-M ignores it and
    recomputes sigma(Z).  Returns (dX, dA, dB, dZ)."""
    X, px = _f64(X)
    A, pa = _f64(A)
    B, pb = _f64(B)
    dY, pdy = _f64(dY)
    Z, pz = _f64(Z)
    n, d_in = X.shape
    r = A.shape[0]
    d_out = B.shape[0]
    m = MODE[mode] if isinstance(mode, str) else int(mode)
    if H is None or m == MODE["cola_m"]:
        ph = None
    else:
        H, ph = _f64(H)
    dX, pdx = _out((n, d_in))
    dA, pda = _out((r, d_in))
    dB, pdb = _out((d_out, r))
    dZ, pdz = _out((n, r))
    lib().oracle_bwd(n, d_in, d_out, r, _sig(sigma), m, int(bool(round_store)), px, pa, pb, pdy,
                     pz, ph, pdx, pda, pdb, pdz)
    return dX, dA, dB, dZ


def recompute_up(Z, B, sigma_kind="silu"):
    """CoLA-M's recompute of a layer output from its saved rank-r activation
    (Sec. 4.2, App. C): H = sigma(Z), Y = H B^T, in the C loops.  Returns
    Y [n x d_out]."""
    Z, pz = _f64(Z)
    B, pb = _f64(B)
    n, r = Z.shape
    d_out = B.shape[0]
    assert B.shape == (d_out, r)
    Y, py = _out((n, d_out))
    lib().oracle_recompute_up(n, d_out, r, _sig(sigma_kind), pz, pb, py)
    return Y


def gate_up_product(Yg, Yu):
    """M = Y_gate * Y_up element-wise (the gated MLP's product, Fig. 4)."""
    Yg, pg = _f64(Yg)
    Yu, pu = _f64(Yu)
    assert Yg.shape == Yu.shape
    M, pm = _out(Yg.shape)
    lib().oracle_gate_up_product(Yg.size, pg, pu, pm)
    return M


def gate_up_backward(dM, Yg, Yu):
    """Gradients of the product: (dY_gate, dY_up) = (dM * Y_up, dM * Y_gate)."""
    dM, pd = _f64(dM)
    Yg, pg = _f64(Yg)
    Yu, pu = _f64(Yu)
    assert dM.shape == Yg.shape == Yu.shape
    dYg, pdg = _out(dM.shape)
    dYu, pdu = _out(dM.shape)
    lib().oracle_gate_up_backward(dM.size, pd, pg, pu, pdg, pdu)
    return dYg, dYu


def gated_fwd(X, Ag, Bg, Au, Bu, sigma="silu", round_store=False):
    """The gate and up layers on one X and their product.  Returns
    (Z_gate, H_gate, Y_gate, Z_up, H_up, Y_up, M)."""
    Zg, Hg, Yg = fwd(X, Ag, Bg, sigma, round_store)
    Zu, Hu, Yu = fwd(X, Au, Bu, sigma, round_store)
    return Zg, Hg, Yg, Zu, Hu, Yu, gate_up_product(Yg, Yu)


def fwd_qkv(X, As, Bs, sigma="silu", round_store=False):
    """Three layers (q, k, v) on one shared X (Fig. 4).  Returns lists (Z, H, Y)."""
    outs = [fwd(X, A, B, sigma, round_store) for A, B in zip(As, Bs)]
    return [o[0] for o in outs], [o[1] for o in outs], [o[2] for o in outs]


def bwd_qkv(X, As, Bs, dYs, Zs, Hs=None, sigma="silu", mode="cola", round_store=False):
    """Backward of three layers sharing X: dX is the sum of the three input
    gradients.  Returns (dX, [dA], [dB], [dZ])."""
    Hs = Hs if Hs is not None else [None] * len(As)
    res = [bwd(X, A, B, dY, Z, H, sigma, mode, round_store)
           for A, B, dY, Z, H in zip(As, Bs, dYs, Zs, Hs)]
    dX = res[0][0].copy()
    for r_ in res[1:]:
        dX += r_[0]
    return dX, [r_[1] for r_ in res], [r_[2] for r_ in res], [r_[3] for r_ in res]


def rows_bf16(X, A, B, rows, dY=None, sigma="silu", round_store=False, d_in=None, d_out=None):
    """Exact Z, H, Y (and dZ, dX when dY is given) on the listed token rows.
    X [n x ld_x] and dY [n x ld_y] are bf16 bits with logical widths d_in, d_out."""
    X, px = _u16(X)
    A, pa = _u16(A)
    B, pb = _u16(B)
    r = A.shape[0]
    d_in = d_in or A.shape[1]
    d_out = d_out or B.shape[0]
    rows, pr = _idx(rows)
    m = rows.size
    Z, pz = _out((m, r))
    H, ph = _out((m, r))
    Y, py = _out((m, d_out))
    dZ, pdz = _out((m, r))
    dX, pdx = _out((m, d_in))
    if dY is not None:
        dY, pdy = _u16(dY)
        ld_y = dY.shape[1]
    else:
        pdy, ld_y = None, 0
    lib().oracle_rows_bf16(d_in, d_out, r, _sig(sigma), int(bool(round_store)), px, X.shape[1],
                           pa, pb, pdy, ld_y, m, pr, pz, ph, py, pdz, pdx)
    if dY is None:
        return Z, H, Y
    return Z, H, Y, dZ, dX


def dA_entries_bf16(X, A, B, dY, ii, kk, sigma="silu", round_store=False, d_out=None):
    X, px = _u16(X)
    A, pa = _u16(A)
    B, pb = _u16(B)
    dY, pdy = _u16(dY)
    r, d_in = A.shape
    d_out = d_out or B.shape[0]
    ii, pi = _idx(ii)
    kk, pk = _idx(kk)
    out, po = _out(ii.shape)
    lib().oracle_dA_entries_bf16(X.shape[0], d_in, d_out, r, _sig(sigma), int(bool(round_store)),
                                 px, X.shape[1], pa, pb, pdy, dY.shape[1], ii.size, pi, pk, po)
    return out


def dB_entries_bf16(X, A, dY, oo, ii, sigma="silu", round_store=False):
    X, px = _u16(X)
    A, pa = _u16(A)
    dY, pdy = _u16(dY)
    r, d_in = A.shape
    oo, po_ = _idx(oo)
    ii, pi = _idx(ii)
    out, po = _out(oo.shape)
    lib().oracle_dB_entries_bf16(X.shape[0], d_in, r, _sig(sigma), int(bool(round_store)), px,
                                 X.shape[1], pa, pdy, dY.shape[1], oo.size, po_, pi, po)
    return out
