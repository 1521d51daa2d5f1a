"""GPU parity of the gated MLP (Fig. 4; Sec. 3.2; App. E) through the C ABI.

Forward, cola_fwd_gate_up: the gate and up CoLA layers read one X, and one
GEMM over both B factors keeps each output tile's gate and up halves in two
accumulators and stores M = Y_gate * Y_up (and Y_gate, Y_up when training).
Backward, cola_bwd_down_gated: the down layer's dX GEMM stores
dY_gate = dM * Y_up and dY_up = dM * Y_gate instead of dM.

Checked against the fp64 oracle (gated_fwd, gate_up_backward, the layer
backward) with the parity tolerance, and bit for bit against the unfused
composition the library's numerics define: M = bf16(Y_gate * Y_up) of the
stored bf16 outputs, dY_gate = bf16(bf16(dM) * Y_up), where the product of
two bf16 values is exact in fp32 and rounded once.  Shapes: ragged token
counts, a d_ff whose rows need a padded pitch (the masked right edge), the
LLaMA-60M widths, and the 1B widths on CTA pairs (sampled).
"""
import numpy as np
import pytest
import torch

import oracle
from cola_helpers import assert_close, make_inputs, padded_empty, padding_intact, to64
from paper_2502_10940_gb300 import inputs as I

pytestmark = pytest.mark.gpu

PAIR, GLU = 4, 32   # launch-trace flags


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()


def _mlp(n, d, d_ff, r, seed):
    from paper_2502_10940_gb300 import cola
    X = make_inputs(n, d, d_ff, r, seed=seed)["X"]
    g = make_inputs(n, d, d_ff, r, seed=seed + 1)
    u = make_inputs(n, d, d_ff, r, seed=seed + 2)
    dn = make_inputs(n, d_ff, d, r, seed=seed + 3)   # the down layer: A [r x d_ff], B [d x r], dY [n x d]
    A_cat = padded_empty(2 * r, d, cola.ld_of(X))
    A_cat.copy_(torch.cat([g["A"], u["A"]], 0))
    return dict(X=X, A_cat=A_cat, Ag=g["A"], Au=u["A"], Bg=g["B"], Bu=u["B"], Ad=dn["A"], Bd=dn["B"], dYd=dn["dY"])


def _forward(t, n, d, d_ff, r, mode):
    from paper_2502_10940_gb300 import cola
    ldf = I.padded_ld(d_ff)
    desc = cola.desc(n, d, d_ff, r, ld_x=cola.ld_of(t["X"]), ld_y=ldf, ld_a=cola.ld_of(t["A_cat"]), sigma="silu",
                     mode=mode)
    ws = cola.workspace(desc, 2)
    train = mode != "infer"
    M = padded_empty(n, d_ff, ldf)
    Yg = padded_empty(n, d_ff, ldf) if train else None
    Yu = padded_empty(n, d_ff, ldf) if train else None
    Z = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda") if train else None
    H = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    with cola.Trace(8) as tr:
        cola.cola_fwd_gate_up(desc, t["X"], t["A_cat"], t["Bg"], t["Bu"], M, Yg, Yu, Z, H, ws)
    assert cola.cola_check_status(ws)[0] == 0
    return dict(M=M, Yg=Yg, Yu=Yu, Z=Z, H=H, desc=desc, ws=ws, trace=tr.records())


def _product_bits(a, b):
    """bf16(a * b) of two bf16 tensors: exact fp32 product, rounded once."""
    return (a.float() * b.float()).to(torch.bfloat16)


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", [(300, 200, 328, 128), (130, 264, 91, 64), (2048, 512, 1376, 128)], ids=str)
def test_gate_up_forward(shape, mode):
    n, d, d_ff, r = shape
    t = _mlp(n, d, d_ff, r, seed=80)
    f = _forward(t, n, d, d_ff, r, mode)
    assert [rec[0] for rec in f["trace"]][-1] == "fwd_glu"
    Zg, Hg, Yg, Zu, Hu, Yu, M = oracle.gated_fwd(to64(t["X"]), to64(t["Ag"]), to64(t["Bg"]), to64(t["Au"]),
                                                 to64(t["Bu"]), "silu")
    assert_close("Y_gate", to64(f["Yg"]), Yg)
    assert_close("Y_up", to64(f["Yu"]), Yu)
    assert_close("M", to64(f["M"]), M)
    assert_close("Z_gate", to64(f["Z"][:, :r]), Zg)
    assert_close("Z_up", to64(f["Z"][:, r:]), Zu)
    if f["H"] is not None:
        assert_close("H_up", to64(f["H"][:, r:]), Hu)
    # the product of the stored outputs, bit for bit; padding untouched
    assert torch.equal(f["M"], _product_bits(f["Yg"], f["Yu"]))
    for k in ("M", "Yg", "Yu"):
        assert padding_intact(f[k], d_ff), k


def test_gate_up_matches_shared_x_outputs_and_inference():
    # the two-accumulator GEMM gives the Y_gate, Y_up of the count-2
    # shared-input forward bit for bit, and the inference forward (M alone) the
    # training forward's M
    from paper_2502_10940_gb300 import cola
    n, d, d_ff, r = 2048, 512, 1376, 128
    t = _mlp(n, d, d_ff, r, seed=81)
    f = _forward(t, n, d, d_ff, r, "cola")
    ldf = I.padded_ld(d_ff)
    Ys = [padded_empty(n, d_ff, ldf) for _ in range(2)]
    desc = f["desc"]
    Z = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, 2 * r), dtype=torch.bfloat16, device="cuda")
    cola.cola_fwd_shared_x(desc, t["X"], t["A_cat"], [t["Bg"], t["Bu"]], Ys, Z, H, f["ws"])
    assert cola.cola_check_status(f["ws"])[0] == 0
    assert torch.equal(Ys[0], f["Yg"]) and torch.equal(Ys[1], f["Yu"])
    fi = _forward(t, n, d, d_ff, r, "infer")
    assert torch.equal(fi["M"], f["M"])


@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", [(300, 200, 328, 128), (130, 264, 91, 64), (2048, 512, 1376, 128)], ids=str)
def test_down_gated_backward(shape, mode):
    from paper_2502_10940_gb300 import cola
    n, d, d_ff, r = shape
    t = _mlp(n, d, d_ff, r, seed=82)
    f = _forward(t, n, d, d_ff, r, "cola")
    ldf = I.padded_ld(d_ff)
    # the down layer on M: forward, then its backward with the gated epilogue
    dd = cola.desc(n, d_ff, d, r, ld_x=ldf, ld_y=cola.ld_of(t["dYd"]), ld_a=cola.ld_of(t["Ad"]), sigma="silu",
                   mode=mode)
    ws = cola.workspace(dd)
    Yd = padded_empty(n, d, cola.ld_of(t["dYd"]))
    Zd = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    Hd = torch.empty((n, r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    cola.cola_fwd(dd, f["M"], t["Ad"], t["Bd"], Yd, Zd, Hd, ws)
    dYg, dYu = padded_empty(n, d_ff, ldf), padded_empty(n, d_ff, ldf)
    dA = padded_empty(r, d_ff, cola.ld_of(t["Ad"]))
    dB = torch.empty((d, r), dtype=torch.bfloat16, device="cuda")
    with cola.Trace(8) as tr:
        cola.cola_bwd_down_gated(dd, f["M"], t["Ad"], t["Bd"], t["dYd"], Zd, Hd, f["Yg"], f["Yu"], dYg, dYu, dA, dB,
                                 ws)
    assert cola.cola_check_status(ws)[0] == 0
    assert any(rec[0] == "bwd_dx" and rec[3] & GLU for rec in tr.records())
    # the plain backward of the same layer gives dM = dX and the same dA, dB
    dM = padded_empty(n, d_ff, ldf)
    dA2, dB2 = padded_empty(r, d_ff, cola.ld_of(t["Ad"])), torch.empty_like(dB)
    cola.cola_bwd(dd, f["M"], t["Ad"], t["Bd"], t["dYd"], Zd, Hd, dM, dA2, dB2, ws)
    assert cola.cola_check_status(ws)[0] == 0
    assert torch.equal(dA, dA2) and torch.equal(dB, dB2)
    assert torch.equal(dYg, _product_bits(dM, f["Yu"]))
    assert torch.equal(dYu, _product_bits(dM, f["Yg"]))
    # against the oracle: the down layer's backward on the same bf16 M, then the product's
    M64, Ad64, Bd64, dY64 = to64(f["M"]), to64(t["Ad"]), to64(t["Bd"]), to64(t["dYd"])
    Zo, Ho, _ = oracle.fwd(M64, Ad64, Bd64, "silu")
    dMo, dAo, dBo, _ = oracle.bwd(M64, Ad64, Bd64, dY64, Zo, Ho, "silu", mode)
    dYgo, dYuo = oracle.gate_up_backward(dMo, to64(f["Yg"]), to64(f["Yu"]))
    assert_close("dY_gate", to64(dYg), dYgo)
    assert_close("dY_up", to64(dYu), dYuo)
    assert_close("dA_down", to64(dA), dAo)
    assert_close("dB_down", to64(dB), dBo)
    assert padding_intact(dYg, d_ff) and padding_intact(dYu, d_ff)


def test_gated_mlp_chain_matches_oracle():
    # the whole gated MLP, forward and backward, through the library: gate/up
    # with the fused product, down on M, down's gated backward, the gate/up
    # backward on dY_gate, dY_up.  Each stage against the oracle fed the
    # library's own bf16 inputs of that stage (the per-layer bound), and the
    # chain's ends against the oracle's all-fp64 chain, where the down layer's
    # input M and the gate/up upstream gradients are themselves bf16 results:
    # two stages of bf16 rounding, so twice the per-layer bound
    from paper_2502_10940_gb300 import cola
    n, d, d_ff, r = 300, 200, 328, 128
    t = _mlp(n, d, d_ff, r, seed=83)
    f = _forward(t, n, d, d_ff, r, "cola")
    ldf = I.padded_ld(d_ff)
    dd = cola.desc(n, d_ff, d, r, ld_x=ldf, ld_y=cola.ld_of(t["dYd"]), ld_a=cola.ld_of(t["Ad"]), sigma="silu")
    wsd = cola.workspace(dd)
    Yd = padded_empty(n, d, cola.ld_of(t["dYd"]))
    Zd = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    Hd = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    cola.cola_fwd(dd, f["M"], t["Ad"], t["Bd"], Yd, Zd, Hd, wsd)
    dYg, dYu = padded_empty(n, d_ff, ldf), padded_empty(n, d_ff, ldf)
    dAd = padded_empty(r, d_ff, cola.ld_of(t["Ad"]))
    dBd = torch.empty((d, r), dtype=torch.bfloat16, device="cuda")
    cola.cola_bwd_down_gated(dd, f["M"], t["Ad"], t["Bd"], t["dYd"], Zd, Hd, f["Yg"], f["Yu"], dYg, dYu, dAd, dBd,
                             wsd)
    dX = padded_empty(n, d, cola.ld_of(t["X"]))
    dA_cat = padded_empty(2 * r, d, cola.ld_of(t["A_cat"]))
    dBs = [torch.empty((d_ff, r), dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    cola.cola_bwd_shared_x(f["desc"], t["X"], t["A_cat"], [t["Bg"], t["Bu"]], [dYg, dYu], f["Z"], f["H"], dX, dA_cat,
                           dBs, f["ws"])
    assert cola.cola_check_status(f["ws"])[0] == 0 and cola.cola_check_status(wsd)[0] == 0
    got = dict(Yd=Yd, dAd=dAd, dBd=dBd, dYg=dYg, dYu=dYu, dX=dX, dAg=dA_cat[:r], dAu=dA_cat[r:], dBg=dBs[0],
               dBu=dBs[1])

    X64 = to64(t["X"])
    Ag, Au, Bg, Bu, Ad, Bd = (to64(t[k]) for k in ("Ag", "Au", "Bg", "Bu", "Ad", "Bd"))
    dYd64 = to64(t["dYd"])

    def chain(M, Yg, Yu, dYg_in=None, dYu_in=None):
        Zdo, Hdo, Ydo = oracle.fwd(M, Ad, Bd, "silu")
        dMo, dAdo, dBdo, _ = oracle.bwd(M, Ad, Bd, dYd64, Zdo, Hdo, "silu", "cola")
        dYgo, dYuo = oracle.gate_up_backward(dMo, Yg, Yu)
        a, b = (dYgo, dYuo) if dYg_in is None else (dYg_in, dYu_in)
        Zg, Hg, _ = oracle.fwd(X64, Ag, Bg, "silu")
        Zu, Hu, _ = oracle.fwd(X64, Au, Bu, "silu")
        dXg, dAg, dBg, _ = oracle.bwd(X64, Ag, Bg, a, Zg, Hg, "silu", "cola")
        dXu, dAu, dBu, _ = oracle.bwd(X64, Au, Bu, b, Zu, Hu, "silu", "cola")
        return dict(Yd=Ydo, dAd=dAdo, dBd=dBdo, dYg=dYgo, dYu=dYuo, dX=dXg + dXu, dAg=dAg, dAu=dAu, dBg=dBg, dBu=dBu)

    # stage by stage: each stage's oracle takes the library's bf16 inputs
    staged = chain(to64(f["M"]), to64(f["Yg"]), to64(f["Yu"]), to64(dYg), to64(dYu))
    for k, v in staged.items():
        assert_close(f"{k} (staged)", to64(got[k]), v)
    # end to end against the all-fp64 chain
    _, _, Ygo, _, _, Yuo, Mo = oracle.gated_fwd(X64, Ag, Bg, Au, Bu, "silu")
    full = chain(Mo, Ygo, Yuo)
    for k, v in full.items():
        assert_close(f"{k} (fp64 chain)", to64(got[k]), v, rel_f=2 * 5e-3, rel_max=2 * 3e-2)


def test_gated_mlp_1b_widths_on_pairs_sampled():
    # d = 2048, d_ff = 5461 (padded pitch 5464, masked right edge), r = 512,
    # 8200 tokens (ragged last pair tile): the product GEMM and the gated dX
    # GEMM on CTA pairs; sampled rows against the oracle, each stage fed the
    # library's own bf16 inputs of that stage
    from paper_2502_10940_gb300 import cola
    n, d, d_ff, r = 8200, 2048, 5461, 512
    t = _mlp(n, d, d_ff, r, seed=84)
    f = _forward(t, n, d, d_ff, r, "cola_m")
    assert f["trace"][-1][0] == "fwd_glu" and f["trace"][-1][3] & PAIR, f["trace"]
    ldf = I.padded_ld(d_ff)
    rows = np.array([0, 1, 127, 128, 4099, n - 257, n - 200, n - 9, n - 1])
    ridx = torch.from_numpy(rows).cuda()

    def bits(x):
        return I.bf16_bits(torch.as_strided(x, (x.shape[0], x.stride(0)), (x.stride(0), 1)))

    Xb = bits(t["X"])
    Zg_o, Hg_o, Yg_o = oracle.rows_bf16(Xb, I.bf16_bits(t["Ag"]), I.bf16_bits(t["Bg"]), rows, None, "silu", d_in=d,
                                        d_out=d_ff)
    Zu_o, Hu_o, Yu_o = oracle.rows_bf16(Xb, I.bf16_bits(t["Au"]), I.bf16_bits(t["Bu"]), rows, None, "silu", d_in=d,
                                        d_out=d_ff)
    assert_close("Y_gate rows", to64(f["Yg"][ridx]), Yg_o)
    assert_close("Y_up rows", to64(f["Yu"][ridx]), Yu_o)
    assert_close("M rows", to64(f["M"][ridx]), oracle.gate_up_product(Yg_o, Yu_o))
    assert torch.equal(f["M"], _product_bits(f["Yg"], f["Yu"]))
    for k in ("M", "Yg", "Yu"):
        assert padding_intact(f[k], d_ff), k

    dd = cola.desc(n, d_ff, d, r, ld_x=ldf, ld_y=cola.ld_of(t["dYd"]), ld_a=cola.ld_of(t["Ad"]), sigma="silu",
                   mode="cola_m")
    ws = cola.workspace(dd)
    Yd = padded_empty(n, d, cola.ld_of(t["dYd"]))
    Zd = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    cola.cola_fwd(dd, f["M"], t["Ad"], t["Bd"], Yd, Zd, None, ws)
    dYg, dYu = padded_empty(n, d_ff, ldf), padded_empty(n, d_ff, ldf)
    dA = padded_empty(r, d_ff, cola.ld_of(t["Ad"]))
    dB = torch.empty((d, r), dtype=torch.bfloat16, device="cuda")
    with cola.Trace(8) as tr:
        cola.cola_bwd_down_gated(dd, f["M"], t["Ad"], t["Bd"], t["dYd"], Zd, None, f["Yg"], f["Yu"], dYg, dYu, dA, dB,
                                 ws)
    assert cola.cola_check_status(ws)[0] == 0
    rec = [x for x in tr.records() if x[0] == "bwd_dx"]
    assert len(rec) == 1 and rec[0][3] & GLU and rec[0][3] & PAIR, tr.records()
    Mb = bits(f["M"])
    _, _, _, _, dM_o = oracle.rows_bf16(Mb, I.bf16_bits(t["Ad"]), I.bf16_bits(t["Bd"]), rows, bits(t["dYd"]), "silu",
                                        d_in=d_ff, d_out=d)
    dYg_o, dYu_o = oracle.gate_up_backward(dM_o, to64(f["Yg"][ridx]), to64(f["Yu"][ridx]))
    assert_close("dY_gate rows", to64(dYg[ridx]), dYg_o)
    assert_close("dY_up rows", to64(dYu[ridx]), dYu_o)
    assert padding_intact(dYg, d_ff) and padding_intact(dYu, d_ff)


@pytest.mark.parametrize("shape", [(8200, 4096, 11008, 1024), (8320, 2048, 5461, 512)], ids=str)
def test_gate_up_256_column_pair_tiles(shape):
    # 7B widths in training (r = 1024) and 1B widths in inference: the product
    # GEMM on 256 x 256 CTA-pair tiles with one TMEM slot whose gate and up
    # accumulators are freed apart.  Sampled rows against the oracle, M the
    # product of the stored outputs bit for bit, and the inference M equal to
    # the training M
    n, d, d_ff, r = shape
    t = _mlp(n, d, d_ff, r, seed=85)
    f = _forward(t, n, d, d_ff, r, "cola_m")
    fi = _forward(t, n, d, d_ff, r, "infer")
    assert f["trace"][-1][0] == "fwd_glu" and f["trace"][-1][3] & PAIR, f["trace"]
    assert fi["trace"][-1][0] == "fwd_glu" and fi["trace"][-1][3] & PAIR, fi["trace"]
    assert torch.equal(fi["M"], f["M"])
    assert torch.equal(f["M"], _product_bits(f["Yg"], f["Yu"]))
    rows = np.array([0, 255, 256, 4097, n - 257, n - 200, n - 1])
    ridx = torch.from_numpy(rows).cuda()

    def bits(x):
        return I.bf16_bits(torch.as_strided(x, (x.shape[0], x.stride(0)), (x.stride(0), 1)))

    Xb = bits(t["X"])
    _, _, Yg_o = oracle.rows_bf16(Xb, I.bf16_bits(t["Ag"]), I.bf16_bits(t["Bg"]), rows, None, "silu", d_in=d,
                                  d_out=d_ff)
    _, _, Yu_o = oracle.rows_bf16(Xb, I.bf16_bits(t["Au"]), I.bf16_bits(t["Bu"]), rows, None, "silu", d_in=d,
                                  d_out=d_ff)
    assert_close("Y_gate rows", to64(f["Yg"][ridx]), Yg_o)
    assert_close("Y_up rows", to64(f["Yu"][ridx]), Yu_o)
    assert_close("M rows", to64(f["M"][ridx]), oracle.gate_up_product(Yg_o, Yu_o))
    for k in ("M", "Yg", "Yu"):
        assert padding_intact(f[k], d_ff), k
    assert padding_intact(fi["M"], d_ff)
