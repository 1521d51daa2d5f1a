"""GPU parity at full workload sizes, in the launch configuration bench.py
times (one layer through cola_fwd / cola_bwd), against the fp64 oracle on
sampled outputs the oracle computes one by one: random token rows of Z, H,
Y and dX (row-local), random entries of dA and dB (each a full reduction
over all n tokens).

The shapes exercise the tile configurations the production workloads select
and the small parity cases do not reach: CTA-pair (cta_group::2) tiles of
compute-heavy launches in every epilogue, including a ragged last pair tile,
the two-sub-tile (256-row) single-CTA tiles, 256-column tiles, ragged widths
with padded pitches (5461 -> 5464), and multi-wave token splits.
"""
import numpy as np
import pytest
import torch

import oracle
from cola_helpers import assert_close, gpu_layer, to64
from paper_2502_10940_gb300 import inputs as I

pytestmark = pytest.mark.gpu

SHAPES = [
    (65536, 2048, 5461, 512),    # LLaMA-1B gate/up: Y with 5461 columns on 256-row tiles
    (65536, 5461, 2048, 512),    # LLaMA-1B down: K = 5461 forward, dA / dX with 5461 columns
    (32768, 8192, 8192, 128),    # r = 128 at 68.7 GFLOP per GEMM: 256-row tiles for Z/H, dZ and dB
    # CTA-pair tiles with a ragged last tile (1B widths, tensor-bound at a few thousand tokens):
    (8320, 2048, 2048, 512),     # the last pair tile's odd CTA holds only rows past the end
    (8200, 2048, 2048, 512),     # the last pair tile ends inside its even CTA's rows
]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()


def _full_bits(t):
    """bf16 bits of the whole padded row-major buffer behind a view."""
    full = torch.as_strided(t, (t.shape[0], t.stride(0)), (t.stride(0), 1))
    return I.bf16_bits(full)


@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_full_size_layer_sampled(shape):
    _check_sampled(shape, "silu", "cola")


# The other activations on the CTA-pair path with a ragged last pair tile, in
# CoLA-M mode: the pair Z/H epilogue applies sigma, the pair dZ epilogue applies
# sigma' and recomputes H = sigma(Z) for dB.
@pytest.mark.parametrize("sigma", ["gelu", "identity"])
def test_pair_tiles_other_activations_cola_m(sigma):
    _check_sampled((8200, 2048, 2048, 512), sigma, "cola_m")


def _check_sampled(shape, sigma, mode):
    n, d_in, d_out, r = shape
    inp = I.layer_inputs(n, d_in, d_out, r, seed=7, device="cuda")
    g = gpu_layer(inp, sigma, mode)
    torch.cuda.synchronize()

    Xb, dYb = _full_bits(inp["X"]), _full_bits(inp["dY"])
    Ab, Bb = I.bf16_bits(inp["A"]), I.bf16_bits(inp["B"])
    rng = np.random.default_rng(1234)
    # random rows plus rows of the last (possibly ragged) 256-row tile
    tail = [n - 1 - k for k in (0, 1, 63, 64, 127, 128, 200) if n - 1 - k >= 0]
    rows = np.unique(np.concatenate([rng.choice(n, 44, replace=False), tail]))
    Z, H, Y, dZ, dX = oracle.rows_bf16(Xb, Ab, Bb, rows, dYb, sigma, d_in=d_in, d_out=d_out)
    ridx = torch.from_numpy(rows).cuda()
    assert_close("Z rows", to64(g["Z"][ridx]), Z)
    if g["H"] is not None:
        assert_close("H rows", to64(g["H"][ridx]), H)
    assert_close("Y rows", to64(g["Y"][ridx]), Y)
    assert_close("dX rows", to64(g["dX"][ridx]), dX)

    ii = rng.integers(0, r, 32)
    kk = rng.integers(0, d_in, 32)
    kk[-1] = d_in - 1
    dA_o = oracle.dA_entries_bf16(Xb, Ab, Bb, dYb, ii, kk, sigma, d_out=d_out)
    dA_g = to64(g["dA"])[ii, kk]
    assert_close("dA entries", dA_g, dA_o)

    oo = rng.integers(0, d_out, 32)
    oo[-1] = d_out - 1
    jj = rng.integers(0, r, 32)
    dB_o = oracle.dB_entries_bf16(Xb, Ab, dYb, oo, jj, sigma)
    dB_g = to64(g["dB"])[oo, jj]
    assert_close("dB entries", dB_g, dB_o)


def test_pair_tiles_cola_m_bitwise_and_fp32_accumulate():
    # On the CTA-pair path (1B widths, ragged last pair tile): CoLA and CoLA-M
    # give the same gradients bit for bit, and fp32 accumulation adds the same
    # gradient onto existing values (sampled against the oracle).
    n, d_in, d_out, r = 8320, 2048, 2048, 512
    inp = I.layer_inputs(n, d_in, d_out, r, seed=9, device="cuda")
    a = gpu_layer(inp, "silu", "cola")
    b = gpu_layer(inp, "silu", "cola_m")
    for k in ["Y", "Z", "dX", "dA", "dB"]:
        assert torch.equal(a[k], b[k]), k
    g0 = torch.Generator(device="cuda").manual_seed(11)
    dA0 = torch.randn((r, d_in), generator=g0, device="cuda")
    dB0 = torch.randn((d_out, r), generator=g0, device="cuda")
    f = gpu_layer(inp, "silu", "cola", wgrad_fp32=True, dA0=dA0, dB0=dB0)
    Xb, dYb = _full_bits(inp["X"]), _full_bits(inp["dY"])
    Ab, Bb = I.bf16_bits(inp["A"]), I.bf16_bits(inp["B"])
    rng = np.random.default_rng(99)
    ii, kk = rng.integers(0, r, 24), rng.integers(0, d_in, 24)
    dA_o = oracle.dA_entries_bf16(Xb, Ab, Bb, dYb, ii, kk, "silu", d_out=d_out)
    assert_close("dA += entries", (to64(f["dA"]) - to64(dA0))[ii, kk], dA_o)
    oo, jj = rng.integers(0, d_out, 24), rng.integers(0, r, 24)
    dB_o = oracle.dB_entries_bf16(Xb, Ab, dYb, oo, jj, "silu")
    assert_close("dB += entries", (to64(f["dB"]) - to64(dB0))[oo, jj], dB_o)
