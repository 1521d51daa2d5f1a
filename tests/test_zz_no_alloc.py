"""cola_wgrad_static_scratch, the weight gradient for callers that cannot
allocate device memory (an operator interface with no workspace argument, or
a process whose device memory is fixed at start-up), checked through the C
ABI against the workspace path cola_bwd, and once directly against the fp64
oracle, on two calls in a row.  The two calls take different inputs, each
checked against its own reference, so that partial sums one call leaves in
the library's one static scratch array cannot make the next call pass.
Collected last on purpose: it shares that array, which must hold no state
that one call leaves for the next.
"""
import numpy as np
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
    for call in range(2):
        inp = make_inputs(n, d_in, d_out, r, seed=21 + call)
        ref = gpu_layer(inp, "silu", "cola")          # dB = dY^T H through cola_bwd (workspace)
        dY, H = inp["dY"], ref["H"]
        dB = torch.full((d_out, r), float("nan"), dtype=torch.bfloat16, device="cuda")
        cola.cola_wgrad_static_scratch(n, d_out, r, dY, cola.ld_of(dY), H, cola.ld_of(H), dB, r)
        torch.cuda.synchronize()
        assert_close(f"dB call {call}", to64(dB), to64(ref["dB"]))


def test_matches_oracle_twice(cola):
    # dA = dZ^T X and dB = dY^T H on the oracle's own dZ and H (fp64, from the
    # same bf16 inputs), through the static scratch with a token split
    import oracle
    n, d_in, d_out, r = 4100, 136, 200, 64
    for call in range(2):
        inp = make_inputs(n, d_in, d_out, r, seed=31 + call)
        X64, A64, B64, dY64 = (to64(inp[k]) for k in ("X", "A", "B", "dY"))
        Z, H, _ = oracle.fwd(X64, A64, B64, "silu")
        dX, dA, dB, dZ = oracle.bwd(X64, A64, B64, dY64, Z, H, "silu", "cola")
        # the GEMM's operands are the bf16 values of the oracle's H and dZ
        Hb = torch.from_numpy(H).to(torch.bfloat16).cuda()
        dZb = torch.from_numpy(dZ).to(torch.bfloat16).cuda()
        out_B = torch.full((d_out, r), float("nan"), dtype=torch.bfloat16, device="cuda")
        cola.cola_wgrad_static_scratch(n, d_out, r, inp["dY"], cola.ld_of(inp["dY"]), Hb, r, out_B, r)
        out_A = torch.full((r, d_in), float("nan"), dtype=torch.float32, device="cuda")
        out_A.zero_()
        cola.cola_wgrad_static_scratch(n, r, d_in, dZb, r, inp["X"], cola.ld_of(inp["X"]), out_A, d_in,
                                       accumulate_f32=True)
        torch.cuda.synchronize()
        assert_close(f"dB call {call}", to64(out_B), dB)
        assert_close(f"dA call {call}", to64(out_A), dA)


def test_fp32_accumulate_twice(cola):
    n, d_in, d_out, r = 300, 200, 328, 128
    refs = []
    acc = torch.zeros((d_out, r), dtype=torch.float32, device="cuda")
    for call in range(2):
        inp = make_inputs(n, d_in, d_out, r, seed=22 + call)
        ref = gpu_layer(inp, "silu", "cola")
        refs.append(to64(ref["dB"]))
        dY, H = inp["dY"], ref["H"]
        cola.cola_wgrad_static_scratch(n, d_out, r, dY, cola.ld_of(dY), H, cola.ld_of(H), acc, r, accumulate_f32=True)
        torch.cuda.synchronize()
        assert_close(f"dB sum after call {call}", to64(acc), np.sum(refs, axis=0))


def test_rejects_problem_beyond_static_scratch(cola):
    t = torch.zeros(64, dtype=torch.bfloat16, device="cuda")
    M = N = 8192                                  # 8192 x 8192 fp32 partials = 256 MiB > 64 MiB
    with pytest.raises(cola.ColaError) as e:
        cola.cola_wgrad_static_scratch(4096, M, N, t, M, t, N, t, N)
    assert e.value.status == 4                    # COLA_ERR_WORKSPACE, before any launch
