"""cola_wgrad_static_scratch, the weight gradient for callers that cannot
allocate device memory (an operator interface with no workspace argument, or
a process whose device memory is fixed at start-up), checked through the C
ABI against the workspace path cola_bwd on the same inputs, on two calls in
a row.  Collected last on purpose: it shares the library's one static
scratch array, which must hold no state that one call leaves for the next.
"""
import pytest
import torch

from cola_helpers import assert_close, gpu_layer, make_inputs, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cola():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()
    from paper_2502_10940_gb300 import cola as c
    return c


# the last shape plans CTA-pair tiles (dB = dY^T H with M = 2048, N = 512 over 65536 tokens)
@pytest.mark.parametrize("shape", [(4100, 136, 200, 64), (2048, 512, 1376, 128), (65536, 2048, 2048, 512)], ids=str)
def test_matches_workspace_path_twice(cola, shape):
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=21)
    ref = gpu_layer(inp, "silu", "cola")          # dB = dY^T H through cola_bwd (workspace)
    dY, H = inp["dY"], ref["H"]
    for call in range(2):
        dB = torch.full((d_out, r), float("nan"), dtype=torch.bfloat16, device="cuda")
        cola.cola_wgrad_static_scratch(n, d_out, r, dY, cola.ld_of(dY), H, cola.ld_of(H), dB, r)
        torch.cuda.synchronize()
        assert_close(f"dB call {call}", to64(dB), to64(ref["dB"]))


def test_fp32_accumulate_twice(cola):
    n, d_in, d_out, r = 300, 200, 328, 128
    inp = make_inputs(n, d_in, d_out, r, seed=22)
    ref = gpu_layer(inp, "silu", "cola")
    dY, H = inp["dY"], ref["H"]
    acc = torch.zeros((d_out, r), dtype=torch.float32, device="cuda")
    for call in range(2):
        cola.cola_wgrad_static_scratch(n, d_out, r, dY, cola.ld_of(dY), H, cola.ld_of(H), acc, r, accumulate_f32=True)
        torch.cuda.synchronize()
        assert_close(f"dB sum after call {call}", to64(acc) / (call + 1), to64(ref["dB"]))


def test_rejects_problem_beyond_static_scratch(cola):
    t = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    M = N = 8192                                  # 8192 x 8192 fp32 partials = 256 MiB > 64 MiB
    with pytest.raises(cola.ColaError) as e:
        cola.cola_wgrad_static_scratch(4096, M, N, t, M, t, N, t, N)
    assert e.value.status == 4                    # COLA_ERR_WORKSPACE, before any launch
