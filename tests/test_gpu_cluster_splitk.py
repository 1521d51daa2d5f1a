"""GPU parity of the cluster-reduced weight gradients: with few output tiles
(a few thousand tokens), dB = dY^T H and dA = dZ^T X split their tokens over
the 2 to 8 CTAs of a thread-block cluster, which add their partial tiles on
chip (each CTA stages its partial and sends every owner its band with one
bulk copy into the owner's shared memory; the owner sums the bands in a fixed
order) and store bf16, or accumulate fp32, in the same launch.  Checked
against the fp64 oracle with the cluster form on and off (off: the planned
split with its reduce launch), on ragged token counts (a ragged last
k-block), ragged and padded gradient widths, cluster sizes that do not
divide the 128 rows of a tile, and fp32 accumulation; that it is
deterministic run to run; and, from the launch trace, that the cluster form
ran (flag bit 7, no reduce launch) where it applies.
"""
import pytest
import torch

from cola_helpers import assert_close, make_inputs, oracle_layer, padded_empty, padding_intact, to64

pytestmark = pytest.mark.gpu

CLUSTER = 128   # trace flag: K split inside thread-block clusters


@pytest.fixture(scope="module")
def cola():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()
    from paper_2502_10940_gb300 import cola as c
    yield c
    c.cola_set_cluster_splitk(True)


def _layer(cola, inp, mode, cluster, wgrad_fp32=False, dA0=None, dB0=None):
    X, A, B, dY = inp["X"], inp["A"], inp["B"], inp["dY"]
    n, d_in = X.shape
    r, d_out = A.shape[0], B.shape[0]
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(X), ld_y=cola.ld_of(dY), ld_a=cola.ld_of(A), sigma="silu",
                  mode=mode, wgrad_fp32=wgrad_fp32)
    ws = cola.workspace(d)
    Y = padded_empty(n, d_out, cola.ld_of(dY))
    Z = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    dX = padded_empty(n, d_in, cola.ld_of(X))
    if wgrad_fp32:
        dA = padded_empty(r, d_in, cola.ld_of(A), torch.float32)
        dA.copy_(dA0)
        dB = dB0.clone()
    else:
        dA = padded_empty(r, d_in, cola.ld_of(A))
        dB = torch.empty((d_out, r), dtype=torch.bfloat16, device="cuda")
    cola.cola_set_cluster_splitk(cluster)
    try:
        with cola.Trace(16) as tr:
            cola.cola_fwd(d, X, A, B, Y, Z, H, ws)
            cola.cola_bwd(d, X, A, B, dY, Z, H, dX, dA, dB, ws)
    finally:
        cola.cola_set_cluster_splitk(True)
    assert cola.cola_check_status(ws)[0] == 0
    recs = [(rec[0], rec[2], rec[3]) for rec in tr.records()]
    return dict(Y=Y, Z=Z, H=H, dX=dX, dA=dA, dB=dB), recs


SHAPES = [
    (2000, 333, 200, 64),      # 2000 tokens (ragged last k-block), dA 64 x 333 (ragged, padded), 5 tiles, 8 splits
    (2048, 512, 512, 128),     # the LLaMA-60M q-proj layer: 8 tiles in clusters of 8
    (1024, 1024, 1024, 256),   # 32 tiles: clusters of 4
    (3000, 512, 1376, 128),    # 15 tiles, 47 k-blocks: clusters of 8 with a short last split
    (1500, 2048, 600, 64),     # 21 tiles, 24 k-blocks: clusters of 6 (bands of 22 rows, the last 18)
    (1800, 2048, 600, 64),     # 21 tiles, 29 k-blocks: clusters of 7 (bands of 19 rows, the last 14)
]


@pytest.mark.parametrize("cluster", [True, False], ids=["cluster", "slabs"])
@pytest.mark.parametrize("mode", ["cola", "cola_m"])
@pytest.mark.parametrize("shape", SHAPES, ids=lambda s: "x".join(map(str, s)))
def test_small_launches_match_oracle(cola, shape, mode, cluster):
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=110)
    g, recs = _layer(cola, inp, mode, cluster)
    o = oracle_layer(inp, "silu", mode)
    for k in ["Y", "Z", "dX", "dA", "dB"] + (["H"] if mode == "cola" else []):
        assert_close(k, to64(g[k]), o[k])
    assert padding_intact(g["Y"], d_out) and padding_intact(g["dX"], d_in)
    clustered = [k for k, _, f in recs if f & CLUSTER]
    assert bool(clustered) == cluster, recs


@pytest.mark.parametrize("shape,S", [((2048, 512, 512, 128), 8), ((1500, 2048, 600, 64), 6),
                                     ((1800, 2048, 600, 64), 7)], ids=str)
def test_cluster_launches_used_where_expected(cola, shape, S):
    n, d_in, d_out, r = shape
    inp = make_inputs(n, d_in, d_out, r, seed=111)
    _, recs = _layer(cola, inp, "cola", True)
    # the backward ends with the weight gradients on clusters of S: no reduce
    # launch after them
    kind, splits, flags = recs[-1]
    assert kind == "wgrad" and flags & CLUSTER and splits == S, recs


def test_cluster_splitk_deterministic(cola):
    inp = make_inputs(2048, 512, 512, 128, seed=112)
    a, _ = _layer(cola, inp, "cola", True)
    b, _ = _layer(cola, inp, "cola", True)
    for k in ("Y", "Z", "H", "dX", "dA", "dB"):
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("cluster", [True, False], ids=["cluster", "slabs"])
def test_cluster_fp32_accumulate(cola, cluster):
    # fp32 weight gradients accumulated onto existing values (D += sum)
    n, d_in, d_out, r = 2048, 512, 512, 128
    inp = make_inputs(n, d_in, d_out, r, seed=113)
    gen = torch.Generator(device="cuda").manual_seed(5)
    dA0 = torch.randn((r, d_in), generator=gen, device="cuda")
    dB0 = torch.randn((d_out, r), generator=gen, device="cuda")
    g, recs = _layer(cola, inp, "cola", cluster, wgrad_fp32=True, dA0=dA0, dB0=dB0)
    o = oracle_layer(inp, "silu", "cola")
    assert_close("dA", to64(g["dA"]) - to64(dA0), o["dA"])
    assert_close("dB", to64(g["dB"]) - to64(dB0), o["dB"])
    assert any(k == "wgrad" and f & CLUSTER for k, _, f in recs) == cluster, recs


def test_set_cluster_splitk_rejects_other_values(cola):
    assert cola.lib().cola_set_cluster_splitk(2) == 1
    assert cola.lib().cola_set_cluster_splitk(-1) == 1
