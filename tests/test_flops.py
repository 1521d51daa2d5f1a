"""FLOP accounting of the CoLA layer pinned to the paper's printed numbers.

Per layer one forward+backward pass is 6 n r (d_in + d_out) (Sec. 3.4's 2MNK
convention and 2x rule); summed over the seven projections of a LLaMA block
it must equal Table 3's CoLA row without the attention score term 12 n^2 d,
and the block ratio to full rank must round to Table 8's printed 0.40.
"""
import os

import pytest

from paper_2502_10940_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_flop_ratios.txt")


def _golden():
    rows = []
    with open(GOLDEN) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append(line.split())
    return rows


@pytest.mark.parametrize("d,d_ff,r", [(512, 1376, 128), (1024, 2736, 256), (2048, 5461, 512),
                                      (4096, 11008, 1024)])
def test_block_sum_equals_table3(d, d_ff, r):
    n = 256
    ours = sum(W.layer_flops(n, l.d_in, l.d_out, l.r) for l in W.llama_block(d, d_ff, r))
    assert ours + 12 * n * n * d == W.paper_flops_cola(n, d, d_ff, r)


def test_printed_ratios_table8():
    n = 256
    seen = 0
    for kind, d, d_ff, r, printed in _golden():
        if kind != "ratio":
            continue
        d, d_ff, r = int(d), int(d_ff), int(r)
        # the projections alone (what the layer replaces; the 12 n^2 d score
        # term is common to both rows) give the printed two-digit ratio ...
        proj = (W.paper_flops_cola(n, d, d_ff, r) - 12 * n * n * d) / (
            W.paper_flops_full_rank(n, d, d_ff) - 12 * n * n * d)
        assert f"{proj:.2f}" == printed
        # ... and with the score term at n = 256 the ratio stays within 0.01 of it
        full = W.paper_flops_cola(n, d, d_ff, r) / W.paper_flops_full_rank(n, d, d_ff)
        assert abs(full - float(printed)) < 0.01
        seen += 1
    assert seen == 2


def test_breakeven_rank_sec34():
    # C_CoLA = C_full with d_ff = 2.5 d (n^2 terms cancel, n -> per-token):
    # r (48 d + 18 * 3.5 d) = 24 d^2 + 45 d^2  =>  r / d = 69 / 111.
    (row,) = [g for g in _golden() if g[0] == "breakeven"]
    d = 10000
    n = 1
    lo, hi = 0.0, float(d)
    for _ in range(100):
        mid = 0.5 * (lo + hi)
        full = 24 * n * d * d + 18 * n * d * 2.5 * d
        cola = 48 * n * d * mid + 18 * n * mid * 3.5 * d
        lo, hi = (mid, hi) if cola < full else (lo, mid)
    assert f"{lo / d:.2f}" == row[4]


def test_workload_flops():
    wl = W.WORKLOADS["60m"]
    assert wl.flops == pytest.approx(4.91e11, rel=2e-3)
    assert W.WORKLOADS["1b"].flops == pytest.approx(7.83e12, rel=2e-3)
    assert W.WORKLOADS["7b"].flops == pytest.approx(1.572e13, rel=2e-3)
    assert W.WORKLOADS["60m-q"].flops == pytest.approx(1.61e9, rel=2e-3)


@pytest.mark.parametrize("name", ["60m", "1b", "7b"])
def test_saved_activations_app_c(name):
    # App. C: CoLA adds 14nr of low-rank activations per block (nr for Ax and
    # nr for sigma(Ax) in each of the 7 layers); CoLA-M keeps 7nr (plus the
    # 2nd of block inputs, which the layers do not hold)
    wl = W.WORKLOADS[name]
    r = wl.layers[0].r
    assert all(l.r == r for l in wl.layers) and len(wl.layers) == 7
    assert W.saved_activation_elems(wl, "cola") == 14 * wl.n * r
    assert W.saved_activation_elems(wl, "cola_m") == 7 * wl.n * r
    assert W.saved_activation_elems(wl, "infer") == 0


@pytest.mark.parametrize("n,d_in,d_out,r", [(2048, 512, 512, 128), (19456, 1376, 512, 64), (300, 200, 328, 128)])
@pytest.mark.parametrize("with_h", [False, True])
def test_fused_launch_accounting_matches_the_two_gemms(n, d_in, d_out, r, with_h):
    # bench.py's algorithmic bytes of a single-kernel pass are those of the two
    # GEMMs it replaces less the rank-r intermediate's round trip (written by
    # the first, read by the second: here it never leaves the chip); the FLOPs
    # are the two GEMMs' FLOPs
    import sys
    sys.path.insert(0, os.path.join(os.path.dirname(__file__), ".."))
    import bench
    e = 2
    # forward: the two-GEMM form always writes Z and H (H kept, or in the
    # workspace to feed F2); the single kernel stores Z, and H only when kept
    fz, ff = bench.launch_cost("fwd_zh", [(n, r, d_in)], 1, 1)
    yz, yf = bench.launch_cost("fwd_y", [(n, d_out, r)], 1, 0)
    fb, fl = bench.launch_cost("fwd_fused", [(n, r, d_in), (n, d_out, r)], 1, (1 if with_h else 0) | 64)
    saved = e * n * r * (1 if with_h else 2)      # H not re-read (and, when not kept, not written)
    assert fb == fz + yz - saved
    assert fl == ff + yf
    # backward: dZ (and H under CoLA-M) stored; dX from dZ on chip
    dz, dzf = bench.launch_cost("bwd_dz", [(n, r, d_out)], 1, 1 if with_h else 0)
    dx, dxf = bench.launch_cost("bwd_dx", [(n, d_in, r)], 1, 0)
    bb, bf = bench.launch_cost("bwd_fused", [(n, r, d_out), (n, d_in, r)], 1, 1 if with_h else 0)
    assert bb == dz + dx - e * n * r
    assert bf == dzf + dxf
