"""GPU parity of the single-kernel backward (Sec. 3.4: dH = dY B, dZ = dH *
sigma'(Z), dX = dZ A, with dZ kept on chip): cola_bwd on a layer with r = 64
or 128 whose dZ and dX GEMMs are HBM-bound, at up to one 128-row tile per SM,
runs dZ and dX in one kernel -- the tile's saved Z loaded into shared memory,
overwritten there by dZ, which the second product reads -- the dX blocks of a
tile shared by several CTAs, and the weight gradients after it.  Checked bit
for bit against the two-GEMM backward (cola_set_fused_backward(0)) in both
training modes and every activation, on ragged token counts, ragged and
padded input widths, a ragged K, a single token and a long stream of tiles;
against the fp64 oracle at the LLaMA-60M shapes; and, from the launch trace,
that the fused kernel is the one that ran.
"""
import numpy as np
import pytest
import torch

from cola_helpers import assert_close, make_inputs, oracle_layer, padded_empty, padding_intact, to64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cola():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()
    from paper_2502_10940_gb300 import cola as c
    yield c
    c.cola_set_fused_backward(True)


def _layer(cola, inp, sigma, mode, fused):
    """Forward, then the backward with the fused form on or off; the
    backward's outputs and the kinds of its launches."""
    X, A, B, dY = inp["X"], inp["A"], inp["B"], inp["dY"]
    n, d_in = X.shape
    r, d_out = A.shape[0], B.shape[0]
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(X), ld_y=cola.ld_of(dY), ld_a=cola.ld_of(A), sigma=sigma,
                  mode=mode)
    ws = cola.workspace(d)
    Y = padded_empty(n, d_out, cola.ld_of(dY))
    Z = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd(d, X, A, B, Y, Z, H, ws)
    dX = padded_empty(n, d_in, cola.ld_of(X))
    dA = padded_empty(r, d_in, cola.ld_of(A))
    dB = torch.full((d_out, r), float("nan"), dtype=torch.bfloat16, device="cuda")
    cola.cola_set_fused_backward(fused)
    try:
        with cola.Trace(8) as tr:
            cola.cola_bwd(d, X, A, B, dY, Z, H, dX, dA, dB, ws)
    finally:
        cola.cola_set_fused_backward(True)
    assert cola.cola_check_status(ws)[0] == 0
    return dict(dX=dX, dA=dA, dB=dB, Z=Z), [rec[0] for rec in tr.records()]


SHAPES = [
    (300, 200, 328, 128),     # ragged n, d_in (2 dX blocks, the second 72 wide) and K = d_out = 328
    (130, 72, 600, 64),       # r = 64
    (200, 91, 333, 128),      # d_in = 91: padded pitch, masked right edge of dX
    (1, 64, 64, 64),          # a single token
    (19456, 1376, 512, 128),  # one tile per SM, the LLaMA-60M down-layer widths: 10.75 dX blocks, one CTA per tile
    (2048, 512, 1376, 128),   # 16 tiles: the 4 dX blocks of a tile on 4 CTAs; K = 1376 (21.5 k-blocks)
]


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_fused_equals_two_gemm_backward(cola, shape, mode):
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=95)
    a, kinds_a = _layer(cola, inp, "silu", mode, True)
    b, kinds_b = _layer(cola, inp, "silu", mode, False)
    assert kinds_a[0] == "bwd_fused" and "bwd_dz" not in kinds_a and "bwd_dx" not in kinds_a, kinds_a
    assert kinds_b[0] == "bwd_dz" and kinds_b[-1] == "bwd_dx", kinds_b
    for k in ("dX", "dA", "dB"):
        assert torch.equal(a[k], b[k]), k
    assert padding_intact(a["dX"], d_in)


@pytest.mark.parametrize("sigma", ["identity", "gelu"])
@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_fused_backward_other_activations(cola, sigma, mode):
    inp = make_inputs(300, 200, 328, 128, seed=96)
    a, _ = _layer(cola, inp, sigma, mode, True)
    b, _ = _layer(cola, inp, sigma, mode, False)
    for k in ("dX", "dA", "dB"):
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_fused_backward_60m_q_matches_oracle(cola, mode):
    # the LLaMA-60M q-proj layer at 2048 tokens, element by element
    inp = make_inputs(2048, 512, 512, 128, seed=97)
    g, kinds = _layer(cola, inp, "silu", mode, True)
    assert kinds[0] == "bwd_fused", kinds
    o = oracle_layer(inp, "silu", mode)
    for k in ("dX", "dA", "dB"):
        assert_close(k, to64(g[k]), o[k])


def test_fused_backward_one_tile_per_sm_sampled_rows(cola):
    # 152 tiles of the LLaMA-60M down-layer widths: dX on sampled rows (the
    # last tile's rows included) against the oracle's exact rows
    import oracle
    from paper_2502_10940_gb300 import inputs as I
    n, d_in, d_out, r = 19456, 1376, 512, 128
    inp = I.layer_inputs(n, d_in, d_out, r, seed=98, device="cuda")
    g, kinds = _layer(cola, inp, "silu", "cola_m", True)
    assert kinds[0] == "bwd_fused", kinds

    def bits(t):
        return I.bf16_bits(torch.as_strided(t, (t.shape[0], t.stride(0)), (t.stride(0), 1)))

    rows = np.unique(np.concatenate([np.random.default_rng(7).choice(n, 24, replace=False), [0, n - 129, n - 1]]))
    _, _, _, _, dX = oracle.rows_bf16(bits(inp["X"]), I.bf16_bits(inp["A"]), I.bf16_bits(inp["B"]), rows,
                                      bits(inp["dY"]), "silu", d_in=d_in, d_out=d_out)
    ridx = torch.from_numpy(rows).cuda()
    assert_close("dX rows", to64(g["dX"][ridx]), dX)


def test_set_fused_backward_rejects_other_values(cola):
    assert cola.lib().cola_set_fused_backward(2) == 1
    assert cola.lib().cola_set_fused_backward(-1) == 1
