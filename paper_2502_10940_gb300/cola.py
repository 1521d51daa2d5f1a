"""Thin ctypes binding of libcola.so (include/cola.h), same names as the C ABI.

Argument marshalling only: tensors become device pointers, the stream
defaults to torch's current CUDA stream, and a non-OK status raises
ColaError.  Every step of the layer runs in the library's kernels; there is
no fallback of any kind -- if libcola.so is missing or cannot load, every
call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libcola.so")

SIGMA = {"identity": 0, "silu": 1, "gelu": 2}
MODE = {"cola": 0, "cola_m": 1, "infer": 2}
STATUS = {0: "COLA_OK", 1: "COLA_ERR_INVALID", 2: "COLA_ERR_ALIGN", 3: "COLA_ERR_UNSUPPORTED",
          4: "COLA_ERR_WORKSPACE", 5: "COLA_ERR_LAUNCH", 6: "COLA_ERR_DEVICE_TIMEOUT"}

# the entry points include/cola.h declares
SYMBOLS = ("cola_workspace_size", "cola_workspace_init", "cola_fwd", "cola_bwd", "cola_fwd_shared_x",
           "cola_bwd_shared_x", "cola_fwd_gate_up", "cola_bwd_down_gated", "cola_recompute_up", "cola_fwd_qkv_fused", "cola_bwd_qkv_fused", "cola_check_status",
           "cola_wgrad_static_scratch", "cola_selftest_wait_timeout", "cola_selftest_wait_timeout_pair",
           "cola_selftest_wait_timeout_cluster",
           "cola_trace_attach", "cola_trace_detach", "cola_set_fused_forward", "cola_set_fused_backward",
           "cola_set_cluster_splitk",
           "cola_status_string")
STATIC_SCRATCH_BYTES = 64 * 1024 * 1024
KERNELS = {0: "fwd_zh", 1: "fwd_y", 2: "bwd_dz", 3: "wgrad", 4: "reduce", 5: "bwd_dx", 6: "sigma", 7: "fwd_glu", 8: "fwd_fused",
           9: "bwd_fused"}


class ColaError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = int(status)
        super().__init__(f"{where}: {STATUS.get(self.status, self.status)} ({_status_text(self.status)})")


class cola_desc_t(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("d_in", ctypes.c_int64), ("d_out", ctypes.c_int64),
                ("r", ctypes.c_int64), ("ld_x", ctypes.c_int64), ("ld_y", ctypes.c_int64),
                ("ld_a", ctypes.c_int64), ("sigma", ctypes.c_int32), ("mode", ctypes.c_int32),
                ("wgrad_fp32", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class cola_trace_slot_t(ctypes.Structure):
    _fields_ = [("start", ctypes.c_void_p), ("stop", ctypes.c_void_p), ("kernel", ctypes.c_int32),
                ("count", ctypes.c_int32), ("mnk", (ctypes.c_int32 * 3) * 4), ("splits", ctypes.c_int32),
                ("flags", ctypes.c_int32)]


_lib = None
_vp = ctypes.c_void_p


def lib():
    """Load libcola.so (once).  Raises if it is missing: there is no fallback."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2502_10940_gb300.build.build()")
        l = ctypes.CDLL(LIB_PATH)
        D = ctypes.POINTER(cola_desc_t)
        st = ctypes.c_int
        l.cola_workspace_size.argtypes = [D, ctypes.c_int32, ctypes.POINTER(ctypes.c_size_t)]
        l.cola_workspace_size.restype = st
        l.cola_workspace_init.argtypes = [_vp, _vp]
        l.cola_workspace_init.restype = st
        l.cola_fwd.argtypes = [D] + [_vp] * 7 + [ctypes.c_size_t, _vp]
        l.cola_fwd.restype = st
        l.cola_bwd.argtypes = [D] + [_vp] * 10 + [ctypes.c_size_t, _vp]
        l.cola_bwd.restype = st
        PP = ctypes.POINTER(ctypes.c_void_p)
        l.cola_fwd_shared_x.argtypes = [D, ctypes.c_int32, _vp, _vp, PP, PP, _vp, _vp, _vp, ctypes.c_size_t, _vp]
        l.cola_fwd_shared_x.restype = st
        l.cola_bwd_shared_x.argtypes = [D, ctypes.c_int32, _vp, _vp, PP, PP, _vp, _vp, _vp, _vp, PP, _vp,
                                        ctypes.c_size_t, _vp]
        l.cola_bwd_shared_x.restype = st
        l.cola_fwd_gate_up.argtypes = [D] + [_vp] * 10 + [ctypes.c_size_t, _vp]
        l.cola_fwd_gate_up.restype = st
        l.cola_bwd_down_gated.argtypes = [D] + [_vp] * 13 + [ctypes.c_size_t, _vp]
        l.cola_bwd_down_gated.restype = st
        l.cola_recompute_up.argtypes = [D, ctypes.c_int32, _vp, PP, PP, _vp, ctypes.c_size_t, _vp]
        l.cola_recompute_up.restype = st
        l.cola_fwd_qkv_fused.argtypes = [D] + [_vp] * 11 + [ctypes.c_size_t, _vp]
        l.cola_fwd_qkv_fused.restype = st
        l.cola_bwd_qkv_fused.argtypes = [D] + [_vp] * 16 + [ctypes.c_size_t, _vp]
        l.cola_bwd_qkv_fused.restype = st
        l.cola_selftest_wait_timeout.argtypes = [_vp, ctypes.c_size_t, _vp]
        l.cola_selftest_wait_timeout.restype = st
        l.cola_selftest_wait_timeout_pair.argtypes = [_vp, ctypes.c_size_t, ctypes.c_int32, _vp]
        l.cola_selftest_wait_timeout_pair.restype = st
        l.cola_selftest_wait_timeout_cluster.argtypes = [_vp, ctypes.c_size_t, _vp]
        l.cola_selftest_wait_timeout_cluster.restype = st
        l.cola_check_status.argtypes = [_vp, _vp, ctypes.POINTER(ctypes.c_uint32)]
        l.cola_check_status.restype = st
        i64 = ctypes.c_int64
        l.cola_wgrad_static_scratch.argtypes = [i64, i64, i64, _vp, i64, _vp, i64, _vp, i64, ctypes.c_int32, _vp]
        l.cola_wgrad_static_scratch.restype = st
        l.cola_trace_attach.argtypes = [ctypes.POINTER(cola_trace_slot_t), ctypes.c_int32,
                                        ctypes.POINTER(ctypes.c_int32)]
        l.cola_trace_attach.restype = st
        l.cola_trace_detach.argtypes = []
        l.cola_trace_detach.restype = st
        l.cola_set_fused_forward.argtypes = [ctypes.c_int32]
        l.cola_set_fused_forward.restype = st
        l.cola_set_fused_backward.argtypes = [ctypes.c_int32]
        l.cola_set_fused_backward.restype = st
        l.cola_set_cluster_splitk.argtypes = [ctypes.c_int32]
        l.cola_set_cluster_splitk.restype = st
        l.cola_status_string.argtypes = [ctypes.c_int]
        l.cola_status_string.restype = ctypes.c_char_p
        _lib = l
    return _lib


def _status_text(status: int) -> str:
    try:
        return lib().cola_status_string(int(status)).decode()
    except Exception:  # noqa: BLE001 -- only used to word an error message
        return "?"


def _check(status: int, where: str):
    if status != 0:
        raise ColaError(status, where)


def desc(n, d_in, d_out, r, ld_x=0, ld_y=0, ld_a=0, sigma="silu", mode="cola", wgrad_fp32=False):
    d = cola_desc_t()
    d.n, d.d_in, d.d_out, d.r = int(n), int(d_in), int(d_out), int(r)
    d.ld_x, d.ld_y, d.ld_a = int(ld_x), int(ld_y), int(ld_a)
    d.sigma = SIGMA[sigma] if isinstance(sigma, str) else int(sigma)
    d.mode = MODE[mode] if isinstance(mode, str) else int(mode)
    d.wgrad_fp32 = int(bool(wgrad_fp32))
    d.reserved = 0
    return d


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(s):
    if s is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _nbytes(ws):
    return ws.numel() * ws.element_size()


def cola_workspace_size(d: cola_desc_t, nproj: int = 1) -> int:
    """Workspace bytes for calls on `nproj` projections sharing one input
    (1: cola_fwd / cola_bwd; 2, 3: the shared-input entry points)."""
    out = ctypes.c_size_t(0)
    _check(lib().cola_workspace_size(ctypes.byref(d), int(nproj), ctypes.byref(out)), "cola_workspace_size")
    return int(out.value)


def cola_workspace_init(ws, stream=None):
    _check(lib().cola_workspace_init(_ptr(ws), _stream(stream)), "cola_workspace_init")


def cola_fwd(d, X, A, B, Y, Z_save, H_save, ws, stream=None):
    _check(lib().cola_fwd(ctypes.byref(d), _ptr(X), _ptr(A), _ptr(B), _ptr(Y), _ptr(Z_save), _ptr(H_save),
                          _ptr(ws), _nbytes(ws), _stream(stream)), "cola_fwd")


def cola_bwd(d, X, A, B, dY, Z_save, H_save, dX, dA, dB, ws, stream=None):
    _check(lib().cola_bwd(ctypes.byref(d), _ptr(X), _ptr(A), _ptr(B), _ptr(dY), _ptr(Z_save), _ptr(H_save),
                          _ptr(dX), _ptr(dA), _ptr(dB), _ptr(ws), _nbytes(ws), _stream(stream)), "cola_bwd")


def _ptr_array(ts):
    arr = (ctypes.c_void_p * len(ts))()
    for i, t in enumerate(ts):
        arr[i] = _ptr(t)
    return arr


def cola_fwd_shared_x(d, X, A_cat, Bs, Ys, Z_cat, H_cat, ws, stream=None):
    _check(lib().cola_fwd_shared_x(ctypes.byref(d), len(Bs), _ptr(X), _ptr(A_cat), _ptr_array(Bs), _ptr_array(Ys),
                                   _ptr(Z_cat), _ptr(H_cat), _ptr(ws), _nbytes(ws), _stream(stream)),
           "cola_fwd_shared_x")


def cola_bwd_shared_x(d, X, A_cat, Bs, dYs, Z_cat, H_cat, dX, dA_cat, dBs, ws, stream=None):
    _check(lib().cola_bwd_shared_x(ctypes.byref(d), len(Bs), _ptr(X), _ptr(A_cat), _ptr_array(Bs), _ptr_array(dYs),
                                   _ptr(Z_cat), _ptr(H_cat), _ptr(dX), _ptr(dA_cat), _ptr_array(dBs), _ptr(ws),
                                   _nbytes(ws), _stream(stream)), "cola_bwd_shared_x")


def cola_fwd_gate_up(d, X, A_cat, B_gate, B_up, M, Y_gate, Y_up, Z_cat, H_cat, ws, stream=None):
    _check(lib().cola_fwd_gate_up(ctypes.byref(d), _ptr(X), _ptr(A_cat), _ptr(B_gate), _ptr(B_up), _ptr(M),
                                  _ptr(Y_gate), _ptr(Y_up), _ptr(Z_cat), _ptr(H_cat), _ptr(ws), _nbytes(ws),
                                  _stream(stream)), "cola_fwd_gate_up")


def cola_bwd_down_gated(d, M, A, B, dY, Z_save, H_save, Y_gate, Y_up, dY_gate, dY_up, dA, dB, ws, stream=None):
    _check(lib().cola_bwd_down_gated(ctypes.byref(d), _ptr(M), _ptr(A), _ptr(B), _ptr(dY), _ptr(Z_save),
                                     _ptr(H_save), _ptr(Y_gate), _ptr(Y_up), _ptr(dY_gate), _ptr(dY_up), _ptr(dA),
                                     _ptr(dB), _ptr(ws), _nbytes(ws), _stream(stream)), "cola_bwd_down_gated")


def cola_recompute_up(d, Z_cat, Bs, Ys, ws, stream=None):
    _check(lib().cola_recompute_up(ctypes.byref(d), len(Bs), _ptr(Z_cat), _ptr_array(Bs), _ptr_array(Ys), _ptr(ws),
                                   _nbytes(ws), _stream(stream)), "cola_recompute_up")


def cola_selftest_wait_timeout(ws, stream=None):
    _check(lib().cola_selftest_wait_timeout(_ptr(ws), _nbytes(ws), _stream(stream)), "cola_selftest_wait_timeout")


def cola_selftest_wait_timeout_pair(ws, variant, stream=None):
    _check(lib().cola_selftest_wait_timeout_pair(_ptr(ws), _nbytes(ws), int(variant), _stream(stream)),
           "cola_selftest_wait_timeout_pair")


def cola_selftest_wait_timeout_cluster(ws, stream=None):
    _check(lib().cola_selftest_wait_timeout_cluster(_ptr(ws), _nbytes(ws), _stream(stream)),
           "cola_selftest_wait_timeout_cluster")


def cola_fwd_qkv_fused(d, X, A_qkv, B_q, B_k, B_v, Y_q, Y_k, Y_v, Z_qkv, H_qkv, ws, stream=None):
    _check(lib().cola_fwd_qkv_fused(ctypes.byref(d), _ptr(X), _ptr(A_qkv), _ptr(B_q), _ptr(B_k), _ptr(B_v),
                                    _ptr(Y_q), _ptr(Y_k), _ptr(Y_v), _ptr(Z_qkv), _ptr(H_qkv), _ptr(ws),
                                    _nbytes(ws), _stream(stream)), "cola_fwd_qkv_fused")


def cola_bwd_qkv_fused(d, X, A_qkv, B_q, B_k, B_v, dY_q, dY_k, dY_v, Z_qkv, H_qkv, dX, dA_qkv, dB_q, dB_k, dB_v,
                       ws, stream=None):
    _check(lib().cola_bwd_qkv_fused(ctypes.byref(d), _ptr(X), _ptr(A_qkv), _ptr(B_q), _ptr(B_k), _ptr(B_v),
                                    _ptr(dY_q), _ptr(dY_k), _ptr(dY_v), _ptr(Z_qkv), _ptr(H_qkv), _ptr(dX),
                                    _ptr(dA_qkv), _ptr(dB_q), _ptr(dB_k), _ptr(dB_v), _ptr(ws), _nbytes(ws),
                                    _stream(stream)), "cola_bwd_qkv_fused")


def cola_check_status(ws, stream=None):
    """Returns (status, raw code); does not raise on a device timeout."""
    code = ctypes.c_uint32(0)
    st = lib().cola_check_status(_ptr(ws), _stream(stream), ctypes.byref(code))
    return int(st), int(code.value)


def cola_set_fused_forward(enable: bool):
    """cola_fwd's single-kernel forward where it applies (default on) or the
    two GEMMs (off), process-wide; the results are the same bit for bit."""
    _check(lib().cola_set_fused_forward(int(bool(enable))), "cola_set_fused_forward")


def cola_set_fused_backward(enable: bool):
    """cola_bwd's single-kernel dZ + dX where it applies (default on) or the
    two GEMMs (off), process-wide; the results are the same bit for bit."""
    _check(lib().cola_set_fused_backward(int(bool(enable))), "cola_set_fused_backward")


def cola_set_cluster_splitk(enable: bool):
    """Weight gradients of few tiles split their tokens inside thread-block
    clusters reduced on chip (default on), or into fp32 slabs with a reduce
    launch (off), process-wide."""
    _check(lib().cola_set_cluster_splitk(int(bool(enable))), "cola_set_cluster_splitk")


def cola_status_string(status: int) -> str:
    return lib().cola_status_string(int(status)).decode()


def cola_wgrad_static_scratch(n_tokens, M, N, P, ld_p, Q, ld_q, D, ld_d, accumulate_f32=False, stream=None):
    """D[M x N] = P[:n_tokens, :M]^T Q[:n_tokens, :N] with the library's static
    device scratch: no workspace, no allocation.  For callers that cannot
    allocate device memory (see include/cola.h)."""
    _check(lib().cola_wgrad_static_scratch(int(n_tokens), int(M), int(N), _ptr(P), int(ld_p), _ptr(Q), int(ld_q),
                                           _ptr(D), int(ld_d), int(bool(accumulate_f32)), _stream(stream)),
           "cola_wgrad_static_scratch")


def cola_trace_attach(slots, capacity: int, count):
    _check(lib().cola_trace_attach(slots, int(capacity), ctypes.byref(count)), "cola_trace_attach")


def cola_trace_detach():
    _check(lib().cola_trace_detach(), "cola_trace_detach")


class Trace:
    """Context manager: while active, every library launch is bracketed by a
    pair of torch CUDA events (timing enabled) recorded on its stream."""

    def __init__(self, capacity: int):
        self.capacity = int(capacity)
        self.events = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                       for _ in range(self.capacity)]
        for a, b in self.events:        # events are created lazily on first record
            a.record()
            b.record()
        self.slots = (cola_trace_slot_t * max(self.capacity, 1))()
        for i, (a, b) in enumerate(self.events):
            self.slots[i].start = a.cuda_event
            self.slots[i].stop = b.cuda_event
        self.count = ctypes.c_int32(0)

    def __enter__(self):
        torch.cuda.synchronize()
        cola_trace_attach(self.slots, self.capacity, self.count)
        return self

    def __exit__(self, *exc):
        cola_trace_detach()
        return False

    def records(self):
        """[(kernel name, [(M, N, K) of each GEMM of the launch], splits, flags, ms)]."""
        torch.cuda.synchronize()
        out = []
        for i in range(self.count.value):
            s_ = self.slots[i]
            a, b = self.events[i]
            shapes = [tuple(int(v) for v in s_.mnk[g]) for g in range(s_.count)]
            out.append((KERNELS.get(s_.kernel, str(s_.kernel)), shapes, s_.splits, s_.flags, a.elapsed_time(b)))
        return out


# ---------------------------------------------------------------- helpers
def ld_of(t) -> int:
    """Row pitch (elements) of a 2-D row-major tensor view."""
    assert t.dim() == 2 and t.stride(1) == 1
    return int(t.stride(0))


def workspace(d: cola_desc_t, nproj: int = 1, device="cuda"):
    """A zero-initialised workspace tensor for `d` (allocated by torch)."""
    nbytes = cola_workspace_size(d, nproj)
    ws = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
    off = (-ws.data_ptr()) % 256
    ws = ws[off:off + nbytes]
    cola_workspace_init(ws)
    return ws
