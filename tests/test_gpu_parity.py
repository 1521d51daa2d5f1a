"""GPU parity: the C-ABI path (tcgen05 kernels) against the fp64 oracle on the
same seeded bf16 inputs, element by element, with the stated tolerance.

Shapes span several 128-row tiles with ragged tails in every dimension
(tokens, d_in, d_out), odd widths whose rows need a padded pitch, ranks that
use both column-tile widths (128, 256), token counts that split the weight
gradient over many CTAs, and the degenerate single-token case.
"""
import numpy as np
import pytest
import torch

from cola_helpers import (assert_close, gpu_layer, make_inputs, oracle_layer, padded_empty, padding_intact,
                          to64)

pytestmark = pytest.mark.gpu

SHAPES = [
    # n,    d_in, d_out, r
    (300, 200, 328, 128),     # ragged n, d_in (k tail), d_out (n-tile tail)
    (257, 520, 136, 256),     # BN=256 rank tile, one-row token tail
    (130, 72, 600, 64),       # rank below one tile width
    (200, 333, 91, 128),      # odd widths -> padded pitches 336 / 96
    (1, 64, 64, 64),          # a single token
    (4100, 136, 200, 64),     # long token reduction: split over 16 CTAs + tail
    (2048, 512, 512, 128),    # LLaMA-60M q-proj layer, n = 2048 (seed 0)
]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
@pytest.mark.parametrize("sigma", ["silu"])
@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_layer_matches_oracle(shape, sigma, mode):
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=0)
    g = gpu_layer(inp, sigma, mode)
    o = oracle_layer(inp, sigma, mode)
    keys = ["Y", "Z", "dX", "dA", "dB"] + (["H"] if mode == "cola" else [])
    for k in keys:
        assert_close(k, to64(g[k]), o[k])
    # the library leaves row padding untouched
    assert padding_intact(g["Y"], d_out) and padding_intact(g["dX"], d_in) and padding_intact(g["dA"], d_in)


@pytest.mark.parametrize("sigma", ["identity", "gelu"])
def test_other_activations(sigma):
    inp = make_inputs(300, 200, 328, 128, seed=1)
    g = gpu_layer(inp, sigma, "cola")
    o = oracle_layer(inp, sigma, "cola")
    for k in ["Y", "Z", "H", "dX", "dA", "dB"]:
        assert_close(k, to64(g[k]), o[k])


def test_storage_rounding_points():
    # Z = bf16(acc) and H = bf16(sigma(bf16 Z)): against the oracle that rounds
    # at the same storage points, Z and H agree to ~1 bf16 ulp.
    inp = make_inputs(300, 200, 328, 128, seed=2)
    g = gpu_layer(inp, "silu", "cola")
    o = oracle_layer(inp, "silu", "cola", round_store=True)
    for k in ["Z", "H"]:
        assert_close(k, to64(g[k]), o[k], rel_f=2e-3, rel_max=1e-2)
    # H is sigma of the stored Z evaluated in fp32 (the logistic to within
    # 1e-4 relative) and rounded once: torch's fp32 SiLU of the stored Z,
    # rounded to bf16, at all but a few elements
    z = g["Z"].float()
    h_ref = (z * torch.sigmoid(z)).to(torch.bfloat16).float()
    mism = (g["H"].float() != h_ref).float().mean().item()
    assert mism < 0.02


@pytest.mark.parametrize("shape", [(300, 200, 328, 128), (4100, 136, 200, 64)], ids=str)
def test_cola_m_gradients_bitwise_equal_cola(shape):
    inp = make_inputs(*shape, seed=3)
    a = gpu_layer(inp, "silu", "cola")
    b = gpu_layer(inp, "silu", "cola_m")
    for k in ["Y", "Z", "dX", "dA", "dB"]:
        assert torch.equal(a[k], b[k]), k


def test_deterministic():
    inp = make_inputs(4100, 136, 200, 64, seed=4)
    a = gpu_layer(inp, "silu", "cola")
    b = gpu_layer(inp, "silu", "cola")
    for k in ["Y", "Z", "H", "dX", "dA", "dB"]:
        assert torch.equal(a[k], b[k]), k


def test_two_host_threads_on_two_streams():
    # The library keeps no per-call host state: two host threads, each with its
    # own stream and workspace, run layers concurrently (their kernels overlap
    # on the GPU) and get the results of a lone run bit for bit.
    import threading
    shapes = [(4100, 136, 200, 64), (2048, 512, 512, 128)]
    inps = [make_inputs(*sh, seed=60 + i) for i, sh in enumerate(shapes)]
    ref = [gpu_layer(inp, "silu", "cola") for inp in inps]
    torch.cuda.synchronize()
    out, err = [None, None], [None, None]

    def work(i):
        try:
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                res = [gpu_layer(inps[i], "silu", "cola") for _ in range(3)]
            s.synchronize()
            out[i] = res
        except Exception as e:  # noqa: BLE001 -- reported by the assertion below
            err[i] = e

    threads = [threading.Thread(target=work, args=(i,)) for i in range(2)]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert err == [None, None], err
    for i in range(2):
        for res in out[i]:
            for k in ["Y", "Z", "H", "dX", "dA", "dB"]:
                assert torch.equal(res[k], ref[i][k]), (i, k)


def test_wgrad_fp32_accumulate():
    n, d_in, d_out, r = 300, 200, 328, 128
    inp = make_inputs(n, d_in, d_out, r, seed=5)
    g0 = torch.Generator(device="cuda").manual_seed(7)
    dA0 = torch.randn((r, d_in), generator=g0, device="cuda")
    dB0 = torch.randn((d_out, r), generator=g0, device="cuda")
    g = gpu_layer(inp, "silu", "cola", wgrad_fp32=True, dA0=dA0, dB0=dB0)
    o = oracle_layer(inp, "silu", "cola")
    assert_close("dA+=", to64(g["dA"]) - to64(dA0), o["dA"])
    assert_close("dB+=", to64(g["dB"]) - to64(dB0), o["dB"])


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", [(300, 200, 64), (2048, 512, 128), (130, 264, 128)], ids=str)
def test_qkv_fused_matches_oracle(shape, mode):
    import oracle
    from paper_2502_10940_gb300 import cola
    from paper_2502_10940_gb300 import inputs as I
    n, d, r = shape
    X = make_inputs(n, d, d, r, seed=10)["X"]
    parts = [make_inputs(n, d, d, r, seed=11 + j) for j in range(3)]
    A_qkv = torch.cat([p["A"] for p in parts], 0)            # [3r x d], dense pitch d
    ldx = cola.ld_of(X)
    A_pad = padded_empty(3 * r, d, ldx)
    A_pad.copy_(A_qkv)
    Bs = [p["B"] for p in parts]
    dYs = [p["dY"] for p in parts]
    ldy = cola.ld_of(dYs[0])
    desc = cola.desc(n, d, d, r, ld_x=ldx, ld_y=ldy, ld_a=ldx, sigma="silu", mode=mode)
    ws = cola.workspace(desc, nproj=3)
    Ys = [padded_empty(n, d, ldy) for _ in range(3)]
    Z = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd_qkv_fused(desc, X, A_pad, *Bs, *Ys, Z, H, ws)
    dX = padded_empty(n, d, ldx)
    dA = padded_empty(3 * r, d, ldx)
    dBs = [torch.empty((d, r), dtype=torch.bfloat16, device="cuda") for _ in range(3)]
    cola.cola_bwd_qkv_fused(desc, X, A_pad, *Bs, *dYs, Z, H, dX, dA, *dBs, ws)
    assert cola.cola_check_status(ws)[0] == 0

    X64 = to64(X)
    As = [to64(p["A"]) for p in parts]
    Zs, Hs, Yo = oracle.fwd_qkv(X64, As, [to64(b) for b in Bs], "silu")
    dXo, dAo, dBo, _ = oracle.bwd_qkv(X64, As, [to64(b) for b in Bs], [to64(t) for t in dYs], Zs, Hs, "silu",
                                      "cola")
    for j in range(3):
        assert_close(f"Y{j}", to64(Ys[j]), Yo[j])
        assert_close(f"Z{j}", to64(Z[:, j * r:(j + 1) * r]), Zs[j])
        if H is not None:
            assert_close(f"H{j}", to64(H[:, j * r:(j + 1) * r]), Hs[j])
        assert_close(f"dB{j}", to64(dBs[j]), dBo[j])
        assert_close(f"dA{j}", to64(dA[j * r:(j + 1) * r]), dAo[j])
    assert_close("dX", to64(dX), dXo)


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_qkv_fused_fp32_accumulate_gelu(mode):
    # fp32 weight gradients through the shared-input backward: dA_qkv [3r x d]
    # and each dB_j are added onto existing fp32 values (micro-batching), with
    # the GELU activation and a ragged token count (a partial last token tile)
    import oracle
    from paper_2502_10940_gb300 import cola
    n, d, r = 1100, 264, 64
    X = make_inputs(n, d, d, r, seed=40)["X"]
    parts = [make_inputs(n, d, d, r, seed=41 + j) for j in range(3)]
    ldx = cola.ld_of(X)
    A_pad = padded_empty(3 * r, d, ldx)
    A_pad.copy_(torch.cat([p["A"] for p in parts], 0))
    Bs = [p["B"] for p in parts]
    dYs = [p["dY"] for p in parts]
    ldy = cola.ld_of(dYs[0])
    desc = cola.desc(n, d, d, r, ld_x=ldx, ld_y=ldy, ld_a=ldx, sigma="gelu", mode=mode, wgrad_fp32=True)
    ws = cola.workspace(desc, nproj=3)
    Ys = [padded_empty(n, d, ldy) for _ in range(3)]
    Z = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd_qkv_fused(desc, X, A_pad, *Bs, *Ys, Z, H, ws)
    g0 = torch.Generator(device="cuda").manual_seed(42)
    dA0 = torch.randn((3 * r, d), generator=g0, device="cuda")
    dB0 = [torch.randn((d, r), generator=g0, device="cuda") for _ in range(3)]
    dX = padded_empty(n, d, ldx)
    dA = padded_empty(3 * r, d, ldx, torch.float32)
    dA.copy_(dA0)
    dBs = [b.clone() for b in dB0]
    cola.cola_bwd_qkv_fused(desc, X, A_pad, *Bs, *dYs, Z, H, dX, dA, *dBs, ws)
    assert cola.cola_check_status(ws)[0] == 0

    X64 = to64(X)
    As = [to64(p["A"]) for p in parts]
    Bo = [to64(b) for b in Bs]
    Zs, Hs, Yo = oracle.fwd_qkv(X64, As, Bo, "gelu")
    dXo, dAo, dBo, _ = oracle.bwd_qkv(X64, As, Bo, [to64(t) for t in dYs], Zs, Hs, "gelu", "cola")
    for j in range(3):
        assert_close(f"dB{j}+=", to64(dBs[j]) - to64(dB0[j]), dBo[j])
        assert_close(f"dA{j}+=", (to64(dA) - to64(dA0))[j * r:(j + 1) * r], dAo[j])
    assert_close("dX", to64(dX), dXo)


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", [(300, 200, 328, 128), (2048, 512, 1376, 128)], ids=str)
def test_shared_x_pair_matches_oracle(shape, mode):
    # gate / up: two projections of one shape reading one X (Fig. 4); dX is
    # the sum of both input gradients, dA_cat one GEMM with M = 2r
    import oracle
    from paper_2502_10940_gb300 import cola
    n, d_in, d_out, r = shape
    X = make_inputs(n, d_in, d_out, r, seed=30)["X"]
    parts = [make_inputs(n, d_in, d_out, r, seed=31 + j) for j in range(2)]
    ldx = cola.ld_of(X)
    A_cat = padded_empty(2 * r, d_in, ldx)
    A_cat.copy_(torch.cat([p["A"] for p in parts], 0))
    Bs = [p["B"] for p in parts]
    dYs = [p["dY"] for p in parts]
    ldy = cola.ld_of(dYs[0])
    desc = cola.desc(n, d_in, d_out, r, ld_x=ldx, ld_y=ldy, ld_a=ldx, sigma="silu", mode=mode)
    ws = cola.workspace(desc, nproj=2)
    Ys = [padded_empty(n, d_out, ldy) for _ in range(2)]
    Z = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd_shared_x(desc, X, A_cat, Bs, Ys, Z, H, ws)
    dX = padded_empty(n, d_in, ldx)
    dA = padded_empty(2 * r, d_in, ldx)
    dBs = [torch.empty((d_out, r), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    cola.cola_bwd_shared_x(desc, X, A_cat, Bs, dYs, Z, H, dX, dA, dBs, ws)
    assert cola.cola_check_status(ws)[0] == 0

    X64 = to64(X)
    As = [to64(p["A"]) for p in parts]
    Bo = [to64(b) for b in Bs]
    Zs, Hs, Yo = oracle.fwd_qkv(X64, As, Bo, "silu")
    dXo, dAo, dBo, _ = oracle.bwd_qkv(X64, As, Bo, [to64(t) for t in dYs], Zs, Hs, "silu", "cola")
    for j in range(2):
        assert_close(f"Y{j}", to64(Ys[j]), Yo[j])
        assert_close(f"Z{j}", to64(Z[:, j * r:(j + 1) * r]), Zs[j])
        assert_close(f"dB{j}", to64(dBs[j]), dBo[j])
        assert_close(f"dA{j}", to64(dA[j * r:(j + 1) * r]), dAo[j])
    assert_close("dX", to64(dX), dXo)
    assert padding_intact(dX, d_in) and padding_intact(Ys[0], d_out)


@pytest.mark.parametrize("shape", [(300, 200, 328, 128), (257, 520, 136, 256), (1, 64, 64, 64)], ids=str)
def test_infer_forward_matches_training_forward(shape):
    # the inference forward stores H alone; Y is bit for bit the training
    # forward's Y (the same kernels round Z, apply sigma and run the Y GEMM),
    # and within tolerance of the oracle
    from paper_2502_10940_gb300 import cola
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=40)
    ref = gpu_layer(inp, "silu", "cola")
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(inp["X"]), ld_y=cola.ld_of(inp["dY"]),
                  ld_a=cola.ld_of(inp["A"]), sigma="silu", mode="infer")
    ws = cola.workspace(d)
    Y = padded_empty(n, d_out, cola.ld_of(inp["dY"]))
    cola.cola_fwd(d, inp["X"], inp["A"], inp["B"], Y, None, None, ws)
    assert cola.cola_check_status(ws)[0] == 0
    assert torch.equal(Y, ref["Y"])
    assert_close("Y", to64(Y), oracle_layer(inp, "silu", "cola")["Y"])
    assert padding_intact(Y, d_out)


def test_infer_shared_x_matches_training_forward():
    from paper_2502_10940_gb300 import cola
    n, d, r = 2048, 512, 128
    X = make_inputs(n, d, d, r, seed=41)["X"]
    parts = [make_inputs(n, d, d, r, seed=42 + j) for j in range(3)]
    ldx = cola.ld_of(X)
    A_cat = padded_empty(3 * r, d, ldx)
    A_cat.copy_(torch.cat([p["A"] for p in parts], 0))
    Bs = [p["B"] for p in parts]
    ldy = cola.ld_of(parts[0]["dY"])
    outs = {}
    for mode in ("cola", "infer"):
        desc = cola.desc(n, d, d, r, ld_x=ldx, ld_y=ldy, ld_a=ldx, sigma="silu", mode=mode)
        ws = cola.workspace(desc, nproj=3)
        Ys = [padded_empty(n, d, ldy) for _ in range(3)]
        Z = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
        H = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
        cola.cola_fwd_shared_x(desc, X, A_cat, Bs, Ys, Z, H, ws)
        assert cola.cola_check_status(ws)[0] == 0
        outs[mode] = Ys
    for a, b in zip(outs["cola"], outs["infer"]):
        assert torch.equal(a, b)


@pytest.mark.parametrize("shape", [(32, 2048, 2048, 512), (100, 512, 1376, 128), (5, 4096, 4096, 1024)], ids=str)
@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_small_n_split_k_forward_and_backward(shape, mode):
    # a few tokens: the forward GEMMs have far fewer tiles than SMs and run
    # split over K (fp32 partials, then the reduce with the Z/H or plain
    # epilogue); forward and backward against the oracle
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=60)
    g = gpu_layer(inp, "silu", mode)
    o = oracle_layer(inp, "silu", mode)
    for k in ["Y", "Z", "dX", "dA", "dB"] + (["H"] if mode == "cola" else []):
        assert_close(k, to64(g[k]), o[k])


def test_small_n_infer_matches_training_forward():
    from paper_2502_10940_gb300 import cola
    n, d_in, d_out, r = 32, 2048, 2048, 512
    inp = make_inputs(n, d_in, d_out, r, seed=61)
    ref = gpu_layer(inp, "silu", "cola")
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(inp["X"]), ld_y=cola.ld_of(inp["dY"]),
                  ld_a=cola.ld_of(inp["A"]), sigma="silu", mode="infer")
    ws = cola.workspace(d)
    Y = padded_empty(n, d_out, cola.ld_of(inp["dY"]))
    cola.cola_fwd(d, inp["X"], inp["A"], inp["B"], Y, None, None, ws)
    assert cola.cola_check_status(ws)[0] == 0
    assert torch.equal(Y, ref["Y"])


@pytest.mark.parametrize("mode", ["cola", "infer"])
def test_small_n_shared_x_split_k(mode):
    # three projections on one X at 40 tokens with K = 1024 in both forward
    # GEMMs: the Z/H GEMM (N = 3r) and the three Y GEMMs run split over K and
    # are finished by the reduce (one Z/H job; three Y jobs in one launch)
    import oracle
    from paper_2502_10940_gb300 import cola
    n, d, r = 40, 1024, 1024
    X = make_inputs(n, d, d, r, seed=70)["X"]
    parts = [make_inputs(n, d, d, r, seed=71 + j) for j in range(3)]
    ldx = cola.ld_of(X)
    A_cat = padded_empty(3 * r, d, ldx)
    A_cat.copy_(torch.cat([p["A"] for p in parts], 0))
    Bs = [p["B"] for p in parts]
    ldy = cola.ld_of(parts[0]["dY"])
    desc = cola.desc(n, d, d, r, ld_x=ldx, ld_y=ldy, ld_a=ldx, sigma="silu", mode=mode)
    ws = cola.workspace(desc, nproj=3)
    Ys = [padded_empty(n, d, ldy) for _ in range(3)]
    Z = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    H = torch.empty((n, 3 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd_shared_x(desc, X, A_cat, Bs, Ys, Z, H, ws)
    assert cola.cola_check_status(ws)[0] == 0
    Zs, Hs, Yo = oracle.fwd_qkv(to64(X), [to64(p["A"]) for p in parts], [to64(b) for b in Bs], "silu")
    for j in range(3):
        assert_close(f"Y{j}", to64(Ys[j]), Yo[j])
        if Z is not None:
            assert_close(f"Z{j}", to64(Z[:, j * r:(j + 1) * r]), Zs[j])
            assert_close(f"H{j}", to64(H[:, j * r:(j + 1) * r]), Hs[j])
        assert padding_intact(Ys[j], d)
