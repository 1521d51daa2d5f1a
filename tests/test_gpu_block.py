"""The block the bench times, on the GPU: what each mode saves (App. C),
CoLA-M's block-level recompute of the up-projections (Sec. 4.2), and the
CUDA-graph replay of a step against the eager launches."""
import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2502_10940_gb300 import build
    build.build()


def _small_block(mode):
    import bench
    from paper_2502_10940_gb300 import workloads as W
    wl = W.Workload("small", 1024, W.llama_block(256, 688, 64), modes=(mode,),
                    phase="infer" if mode == "infer" else "train")
    return wl, bench.Block(wl, mode, "cuda:0", seed=3)


@pytest.mark.parametrize("mode", ["cola", "cola_m", "infer"])
def test_saved_activations_match_app_c(mode):
    from paper_2502_10940_gb300 import workloads as W
    wl, blk = _small_block(mode)
    kept = sum(g[k].numel() for g in blk.groups for k in ("Z", "H") if g.get(k) is not None)
    assert kept == W.saved_activation_elems(wl, mode)


def test_recompute_up_reproduces_block_outputs():
    # CoLA-M forward, then Y_j = sigma(Z_j) B_j^T from the saved Z of every
    # group: bit for bit the forward's outputs
    from paper_2502_10940_gb300 import cola
    wl, blk = _small_block("cola_m")
    blk.forward()
    torch.cuda.synchronize()
    saved = [[s["Y"].clone() for s in g["members"]] for g in blk.groups]
    for g in blk.groups:
        for s in g["members"]:
            s["Y"].zero_()
    for g in blk.groups:
        m = g["members"]
        cola.cola_recompute_up(g["desc"], g["Z"], [s["B"] for s in m], [s["Y"] for s in m], blk.ws)
    blk.check()
    for g, ys in zip(blk.groups, saved):
        for s, y in zip(g["members"], ys):
            assert torch.equal(s["Y"], y)


def test_recompute_up_matches_oracle():
    import oracle
    from cola_helpers import assert_close, make_inputs, padded_empty, to64
    from paper_2502_10940_gb300 import cola
    n, d_in, d_out, r = 300, 200, 328, 128
    inp = make_inputs(n, d_in, d_out, r, seed=50)
    ldy = cola.ld_of(inp["dY"])
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(inp["X"]), ld_y=ldy, ld_a=cola.ld_of(inp["A"]),
                  sigma="silu", mode="cola_m")
    ws = cola.workspace(d)
    Z = (torch.randn((n, r), device="cuda") * 2).to(torch.bfloat16)
    Y = padded_empty(n, d_out, ldy)
    cola.cola_recompute_up(d, Z, [inp["B"]], [Y], ws)
    assert cola.cola_check_status(ws)[0] == 0
    assert_close("Y", to64(Y), oracle.recompute_up(to64(Z), to64(inp["B"]), "silu"))


@pytest.mark.parametrize("mode", ["cola", "infer"])
def test_graph_replay_equals_eager(mode):
    wl, blk = _small_block(mode)
    blk.step()
    torch.cuda.synchronize()
    outs = [t.clone() for t in blk.step_results()]
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        blk.step()
    for t in blk.step_results():
        t.zero_()
    g.replay()
    torch.cuda.synchronize()
    blk.check()
    for a, b in zip(outs, blk.step_results()):
        assert torch.equal(a, b)
