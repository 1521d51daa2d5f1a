"""Failure detection on the GPU without a fault: a kernel whose wait can never
be satisfied (its TMA producer issues nothing) gives up after its 2 s bound,
records the timeout in the workspace status word and exits; the host reads
COLA_ERR_DEVICE_TIMEOUT, and the context keeps working."""
import time

import pytest
import torch

from cola_helpers import assert_close, gpu_layer, make_inputs, oracle_layer, to64

pytestmark = pytest.mark.gpu

MMA, EPILOGUE = 0x2, 0x4


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()


def test_wait_runs_out_and_is_reported():
    from paper_2502_10940_gb300 import cola
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    cola.cola_workspace_init(ws)
    assert cola.cola_check_status(ws)[0] == 0
    t0 = time.perf_counter()
    cola.cola_selftest_wait_timeout(ws)
    st, code = cola.cola_check_status(ws)
    dt = time.perf_counter() - t0
    assert st == 6  # COLA_ERR_DEVICE_TIMEOUT
    assert code & MMA and not code & ~(MMA | EPILOGUE), hex(code)
    assert 1.5 < dt < 30.0
    # the check cleared the word, and nothing past it was touched
    assert cola.cola_check_status(ws)[0] == 0
    assert int(ws[256:].count_nonzero()) == 0
    # the context still runs the layer correctly
    inp = make_inputs(300, 200, 328, 128, seed=21)
    g = gpu_layer(inp, "silu", "cola")
    o = oracle_layer(inp, "silu", "cola")
    for k in ["Y", "dX", "dA", "dB"]:
        assert_close(k, to64(g[k]), o[k])


def test_selftest_argument_errors():
    from paper_2502_10940_gb300 import cola
    lib = cola.lib()
    assert lib.cola_selftest_wait_timeout(None, 1 << 20, None) == 1
    ws = torch.zeros(1024, dtype=torch.uint8, device="cuda")
    assert lib.cola_selftest_wait_timeout(ws.data_ptr(), ws.numel(), None) == 4   # too small
