"""Host-side checks of the C ABI that need no GPU: the library builds and
loads, exports every entry point include/cola.h declares, and rejects bad
arguments before it touches a device (every call below returns during
argument validation; no pointer is ever dereferenced)."""
import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "cola.h")


@pytest.fixture(scope="module")
def L():
    from paper_2502_10940_gb300 import build as B
    if not os.path.exists(B.LIB):
        if shutil.which(B.nvcc()) is None and not os.path.exists(B.nvcc()):
            pytest.skip("nvcc not available to build libcola.so")
        B.build()
    from paper_2502_10940_gb300 import cola
    return cola


def _declared():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"^(?:cola_status_t|const char\*)\s+(cola_\w+)\s*\(", text, re.M)))


def test_header_declares_the_entry_points(L):
    assert _declared() == sorted(L.SYMBOLS)


def test_library_exports_every_declared_symbol(L):
    raw = ctypes.CDLL(L.LIB_PATH)
    for name in _declared():
        assert hasattr(raw, name), name


def test_status_strings(L):
    for code in range(7):
        assert L.cola_status_string(code)
    assert "unknown" in L.cola_status_string(99)


def test_desc_layout_matches_header(L):
    # 7 int64 + 4 int32, no padding
    assert ctypes.sizeof(L.cola_desc_t) == 7 * 8 + 4 * 4


def _ws_size(L, d, nproj=1):
    out = ctypes.c_size_t(0)
    return L.lib().cola_workspace_size(ctypes.byref(d), nproj, ctypes.byref(out))


@pytest.mark.parametrize("kw,code", [
    (dict(r=100), 3),                    # r not a multiple of 64 -> UNSUPPORTED
    (dict(r=0), 1),
    (dict(n=0), 1),
    (dict(d_in=-3), 1),
    (dict(ld_x=100), 1),                  # pitch below the width
    (dict(ld_y=132), 1),                  # pitch not a multiple of 8
    (dict(sigma=7), 1),
    (dict(mode=5), 1),
    (dict(n=1 << 30, d_in=1 << 20, d_out=1 << 20, r=128), 3),   # more work units than 32 bits number
])
def test_workspace_size_rejects_bad_desc(L, kw, code):
    args = dict(n=256, d_in=128, d_out=128, r=64)
    args.update({k: v for k, v in kw.items() if k in args})
    extra = {k: v for k, v in kw.items() if k not in args}
    d = L.desc(**args, **extra)
    assert _ws_size(L, d) == code


def test_workspace_size_rejects_null_out_and_bad_nproj(L):
    d = L.desc(256, 128, 128, 64)
    assert L.lib().cola_workspace_size(ctypes.byref(d), 1, None) == 1
    out = ctypes.c_size_t(0)
    assert L.lib().cola_workspace_size(ctypes.byref(d), 0, ctypes.byref(out)) == 1
    assert L.lib().cola_workspace_size(ctypes.byref(d), 4, ctypes.byref(out)) == 1
    assert L.lib().cola_workspace_size(None, 1, ctypes.byref(out)) == 1


FAKE = 0x100000  # 16-byte aligned, never dereferenced


def test_fwd_argument_errors(L):
    f = L.lib().cola_fwd
    d = L.desc(256, 128, 128, 64, mode="cola")
    # null input
    assert f(ctypes.byref(d), None, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    # misaligned input
    assert f(ctypes.byref(d), FAKE + 2, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 2
    # CoLA needs H_save
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20, None) == 1
    # CoLA-M forbids H_save
    dm = L.desc(256, 128, 128, 64, mode="cola_m")
    assert f(ctypes.byref(dm), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1
    # bad rank
    db = L.desc(256, 128, 128, 96)
    assert f(ctypes.byref(db), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 3
    d.reserved = 1
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1


def test_bwd_argument_errors(L):
    f = L.lib().cola_bwd
    d = L.desc(256, 128, 128, 64, mode="cola_m")
    ok = [FAKE] * 10
    args = list(ok)
    args[5] = FAKE  # H_save given under CoLA-M
    assert f(ctypes.byref(d), *args, 1 << 20, None) == 1
    args = list(ok)
    args[5] = None
    args[7] = FAKE + 8  # misaligned dA
    assert f(ctypes.byref(d), *args, 1 << 20, None) == 2
    args[7] = None      # null dA
    assert f(ctypes.byref(d), *args, 1 << 20, None) == 1


def test_qkv_argument_errors(L):
    d = L.desc(256, 128, 128, 64, mode="cola")
    f = L.lib().cola_fwd_qkv_fused
    args = [FAKE] * 11
    args[3] = None  # B_k missing
    assert f(ctypes.byref(d), *args, 1 << 20, None) == 1
    g = L.lib().cola_bwd_qkv_fused
    args = [FAKE] * 16
    args[13] = FAKE + 4  # misaligned dB_k
    assert g(ctypes.byref(d), *args, 1 << 20, None) == 2


def test_shared_x_argument_errors(L):
    d = L.desc(256, 128, 128, 64, mode="cola")
    f = L.lib().cola_fwd_shared_x
    ok2 = (ctypes.c_void_p * 2)(FAKE, FAKE)
    bad = (ctypes.c_void_p * 2)(FAKE, FAKE + 4)
    nul = (ctypes.c_void_p * 2)(FAKE, None)
    assert f(ctypes.byref(d), 1, FAKE, FAKE, ok2, ok2, FAKE, FAKE, FAKE, 1 << 20, None) == 1   # count < 2
    assert f(ctypes.byref(d), 4, FAKE, FAKE, ok2, ok2, FAKE, FAKE, FAKE, 1 << 20, None) == 1   # count > 3
    assert f(ctypes.byref(d), 2, FAKE, FAKE, nul, ok2, FAKE, FAKE, FAKE, 1 << 20, None) == 1   # null B[1]
    assert f(ctypes.byref(d), 2, FAKE, FAKE, ok2, bad, FAKE, FAKE, FAKE, 1 << 20, None) == 2   # misaligned Y[1]
    assert f(ctypes.byref(d), 2, FAKE, FAKE, None, ok2, FAKE, FAKE, FAKE, 1 << 20, None) == 1  # no B array
    g = L.lib().cola_bwd_shared_x
    dm = L.desc(256, 128, 128, 64, mode="cola_m")
    assert g(ctypes.byref(dm), 2, FAKE, FAKE, ok2, ok2, FAKE, FAKE, FAKE, FAKE, ok2, FAKE, 1 << 20, None) == 1  # H under CoLA-M
    assert g(ctypes.byref(dm), 2, FAKE, FAKE, ok2, ok2, FAKE, None, FAKE, FAKE, bad, FAKE, 1 << 20, None) == 2


def test_infer_mode_argument_errors(L):
    d = L.desc(256, 128, 128, 64, mode="infer")
    f = L.lib().cola_fwd
    # inference saves nothing: Z_save and H_save must both be NULL
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20, None) == 1
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, 1 << 20, None) == 1
    # the backward entry points reject the inference mode
    assert L.lib().cola_bwd(ctypes.byref(d), *([FAKE] * 5), None, *([FAKE] * 4), 1 << 20, None) == 1
    ok2 = (ctypes.c_void_p * 2)(FAKE, FAKE)
    assert L.lib().cola_bwd_shared_x(ctypes.byref(d), 2, FAKE, FAKE, ok2, ok2, FAKE, None, FAKE, FAKE, ok2, FAKE,
                                     1 << 20, None) == 1
    # a training-mode forward still needs Z_save
    dc = L.desc(256, 128, 128, 64, mode="cola_m")
    assert f(ctypes.byref(dc), FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 20, None) == 1


def test_gated_mlp_argument_errors(L):
    # cola_fwd_gate_up(desc, X, A_cat, B_gate, B_up, M, Y_gate, Y_up, Z_cat, H_cat, ws, ws_bytes, stream)
    f = L.lib().cola_fwd_gate_up
    d = L.desc(256, 128, 344, 64, mode="cola")
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1  # no M
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 1  # training needs Y_gate
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE + 2, FAKE, FAKE, FAKE, 1 << 20, None) == 2
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE + 8, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None) == 2
    assert f(ctypes.byref(d), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, 1 << 20, None) == 1  # CoLA saves H
    di = L.desc(256, 128, 344, 64, mode="infer")
    assert f(ctypes.byref(di), FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, FAKE, None, None, FAKE, 1 << 20, None) == 1  # inference: no Y_gate
    assert f(ctypes.byref(L.desc(256, 128, 344, 100)), *([FAKE] * 10), 1 << 20, None) == 3   # r % 64
    # cola_bwd_down_gated(desc, M, A, B, dY, Z, H, Y_gate, Y_up, dY_gate, dY_up, dA, dB, ws, ws_bytes, stream)
    g = L.lib().cola_bwd_down_gated
    dd = L.desc(256, 344, 128, 64, ld_x=352, mode="cola_m")
    assert g(ctypes.byref(dd), *([FAKE] * 5), FAKE, *([FAKE] * 7), 1 << 20, None) == 1                # H under CoLA-M
    assert g(ctypes.byref(dd), *([FAKE] * 5), None, FAKE, None, *([FAKE] * 5), 1 << 20, None) == 1    # no Y_up
    assert g(ctypes.byref(dd), *([FAKE] * 5), None, FAKE, FAKE, FAKE + 4, *([FAKE] * 4), 1 << 20, None) == 2
    assert g(ctypes.byref(L.desc(256, 344, 128, 64, mode="infer")), *([FAKE] * 5), None, *([FAKE] * 7), 1 << 20,
             None) == 1                                                                               # no backward in inference


def test_selftest_argument_errors(L):
    f = L.lib().cola_selftest_wait_timeout
    assert f(None, 1 << 20, None) == 1
    assert f(FAKE + 16, 1 << 20, None) == 2      # not 256-byte aligned
    assert f(FAKE, 1024, None) == 4              # smaller than the status word plus three tiles


def test_pair_selftest_argument_errors(L):
    f = L.lib().cola_selftest_wait_timeout_pair
    assert f(None, 1 << 20, 1, None) == 1
    assert f(FAKE, 1 << 20, 0, None) == 1        # no such variant
    assert f(FAKE, 1 << 20, 3, None) == 1
    assert f(FAKE + 16, 1 << 20, 1, None) == 2   # not 256-byte aligned
    assert f(FAKE, 4096, 2, None) == 4           # smaller than the status word plus the operands


def test_cluster_selftest_argument_errors(L):
    f = L.lib().cola_selftest_wait_timeout_cluster
    assert f(None, 1 << 20, None) == 1
    assert f(FAKE + 16, 1 << 20, None) == 2      # not 256-byte aligned
    assert f(FAKE, 4096, None) == 4              # smaller than the status word plus the operands


@pytest.mark.parametrize("name", ["cola_set_fused_forward", "cola_set_fused_backward", "cola_set_cluster_splitk"])
def test_set_fused_argument_errors(L, name):
    f = getattr(L.lib(), name)
    assert f(2) == 1 and f(-1) == 1
    assert f(1) == 0                             # the default, restored


def test_workspace_init_and_check_reject_null(L):
    assert L.lib().cola_workspace_init(None, None) == 1
    assert L.lib().cola_workspace_init(FAKE + 16, None) == 2   # not 256-byte aligned
    assert L.lib().cola_check_status(None, None, None) == 1
