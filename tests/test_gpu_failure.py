"""Failure detection on the GPU without a fault: a kernel whose wait can never
be satisfied (its TMA producer issues nothing) gives up after its 2 s bound,
records the timeout in the workspace status word and exits; the host reads
COLA_ERR_DEVICE_TIMEOUT, and the context keeps working.  The same on a CTA
pair, where the odd CTA's loads complete on the even CTA's barriers: with no
loads at all, and with the odd CTA stopping after one k-block while the even
CTA's loads of later stages land, in which case the pair's abort drain must
see every load of both CTAs land (no drain-timeout bit) before it exits.  And
on a cluster-reduced weight gradient, where one CTA of the cluster gives up on
its main loop: it still sends its (zero) partial band, the other CTA
completes, and the exchange between them ends without a drain timeout."""
import time

import pytest
import torch

from cola_helpers import assert_close, gpu_layer, make_inputs, oracle_layer, to64

pytestmark = pytest.mark.gpu

PRODUCER, MMA, EPILOGUE, DRAIN = 0x1, 0x2, 0x4, 0x8
PAIR = 4   # launch-trace flag: the GEMM ran on CTA pairs
CLUSTER = 128   # launch-trace flag: the token splits were reduced inside a cluster


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


@pytest.mark.parametrize("variant", [1, 2], ids=["no-loads", "odd-stops-after-one-kblock"])
def test_pair_wait_runs_out_and_drains(variant):
    import numpy as np

    import oracle
    from paper_2502_10940_gb300 import cola
    from paper_2502_10940_gb300 import inputs as I
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    cola.cola_workspace_init(ws)
    assert cola.cola_check_status(ws)[0] == 0
    t0 = time.perf_counter()
    with cola.Trace(4) as tr:
        cola.cola_selftest_wait_timeout_pair(ws, variant)
    st, code = cola.cola_check_status(ws)
    dt = time.perf_counter() - t0
    recs = tr.records()
    assert len(recs) == 1 and recs[0][3] & PAIR, recs
    assert st == 6  # COLA_ERR_DEVICE_TIMEOUT
    assert code & (PRODUCER | MMA | EPILOGUE), hex(code)
    assert not code & ~(PRODUCER | MMA | EPILOGUE), hex(code)   # in particular no drain timeout
    assert 1.5 < dt < 30.0
    assert cola.cola_check_status(ws)[0] == 0
    assert int(ws[256:].count_nonzero()) == 0    # operands only read, nothing stored
    # the context still runs a layer on CTA pairs correctly (1B widths, ragged last pair tile)
    n, d_in, d_out, r = 8200, 2048, 2048, 512
    inp = I.layer_inputs(n, d_in, d_out, r, seed=13, device="cuda")
    with cola.Trace(16) as tr:
        g = gpu_layer(inp, "silu", "cola")
    assert all(rec[3] & PAIR for rec in tr.records() if rec[0] != "reduce")

    def bits(t):
        return I.bf16_bits(torch.as_strided(t, (t.shape[0], t.stride(0)), (t.stride(0), 1)))

    Xb, dYb, Ab, Bb = bits(inp["X"]), bits(inp["dY"]), I.bf16_bits(inp["A"]), I.bf16_bits(inp["B"])
    rows = np.array([0, 1, 4097, n - 200, n - 9, n - 1])
    Z, H, Y, dZ, dX = oracle.rows_bf16(Xb, Ab, Bb, rows, dYb, "silu", d_in=d_in, d_out=d_out)
    ridx = torch.from_numpy(rows).cuda()
    for name, got, ref in (("Z", g["Z"], Z), ("H", g["H"], H), ("Y", g["Y"], Y), ("dX", g["dX"], dX)):
        assert_close(name, to64(got[ridx]), ref)
    ii, kk = np.array([0, 7, r - 1]), np.array([3, 1000, d_in - 1])
    assert_close("dA", to64(g["dA"])[ii, kk],
                 oracle.dA_entries_bf16(Xb, Ab, Bb, dYb, ii, kk, "silu", round_store=True, d_out=d_out))
    oo, jj = np.array([5, 1500, d_out - 1]), np.array([0, 200, r - 1])
    assert_close("dB", to64(g["dB"])[oo, jj], oracle.dB_entries_bf16(Xb, Ab, dYb, oo, jj, "silu", round_store=True))


def test_pair_selftest_argument_errors():
    from paper_2502_10940_gb300 import cola
    lib = cola.lib()
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    assert lib.cola_selftest_wait_timeout_pair(None, 1 << 20, 1, None) == 1
    assert lib.cola_selftest_wait_timeout_pair(ws.data_ptr(), ws.numel(), 3, None) == 1    # no such variant
    assert lib.cola_selftest_wait_timeout_pair(ws.data_ptr(), 4096, 1, None) == 4          # too small


def test_cluster_wait_runs_out_and_exchange_completes():
    from paper_2502_10940_gb300 import cola
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    cola.cola_workspace_init(ws)
    assert cola.cola_check_status(ws)[0] == 0
    t0 = time.perf_counter()
    with cola.Trace(4) as tr:
        cola.cola_selftest_wait_timeout_cluster(ws)
    st, code = cola.cola_check_status(ws)
    dt = time.perf_counter() - t0
    recs = tr.records()
    assert len(recs) == 1 and recs[0][3] & CLUSTER and recs[0][2] == 2, recs
    assert st == 6  # COLA_ERR_DEVICE_TIMEOUT
    assert code & (PRODUCER | MMA | EPILOGUE), hex(code)
    assert not code & ~(PRODUCER | MMA | EPILOGUE), hex(code)   # the exchange completed: no drain timeout
    assert 1.5 < dt < 30.0
    assert cola.cola_check_status(ws)[0] == 0
    # the context still runs cluster-reduced weight gradients correctly
    inp = make_inputs(2048, 512, 512, 128, seed=23)
    with cola.Trace(16) as tr:
        g = gpu_layer(inp, "silu", "cola")
    assert any(rec[0] == "wgrad" and rec[3] & CLUSTER for rec in tr.records()), tr.records()
    o = oracle_layer(inp, "silu", "cola")
    for k in ["Y", "dX", "dA", "dB"]:
        assert_close(k, to64(g[k]), o[k])
