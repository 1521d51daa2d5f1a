"""Layer shapes of the LLaMA-style CoLA blocks and their FLOP accounting.

Every full-size projection of a LLaMA decoder block -- q, k, v, o of the
attention and gate, up, down of the MLP -- becomes one CoLA auto-encoder
layer h = B sigma(A x) (Sec. 3.2, Fig. 4).  FLOPs follow the paper's
2MNK convention with elementwise work left out (Sec. 3.4): per layer the
forward is 2 n r (d_in + d_out) and the backward twice that, so one
forward+backward pass costs 6 n r (d_in + d_out).  Summed over a block this
is the paper's 48ndr + 18nr(d + d_ff) (Table 3); the attention score term
12 n^2 d is not part of the layer and is not counted.
"""
from __future__ import annotations

from dataclasses import dataclass, field


@dataclass(frozen=True)
class Layer:
    name: str
    d_in: int
    d_out: int
    r: int
    x: str  # name of the input activation this layer reads (shared X => same name)


@dataclass(frozen=True)
class Workload:
    name: str
    n: int                  # tokens (sequences x sequence length)
    layers: tuple
    modes: tuple = ("cola",)
    fused_qkv: bool = True
    desc: str = ""
    seqs: int = 0
    seq_len: int = 256
    phase: str = "train"    # "train": forward + backward; "infer": forward only, nothing saved
    # the MLP as LLaMA wires it (Fig. 4): the down layer reads M = Y_gate * Y_up,
    # formed in the gate/up output GEMM, and its backward hands dY_gate, dY_up
    # to the gate/up backward; otherwise the down input and the gate/up
    # upstream gradients are independent synthetic tensors
    gated: bool = False

    @property
    def flops(self) -> float:
        f = fwd_flops if self.phase == "infer" else layer_flops
        return float(sum(f(self.n, l.d_in, l.d_out, l.r) for l in self.layers))


def layer_flops(n: int, d_in: int, d_out: int, r: int) -> int:
    """fwd 2nr(d_in+d_out) + bwd 4nr(d_in+d_out) (Sec. 3.4, App. B)."""
    return 6 * n * r * (d_in + d_out)


def fwd_flops(n: int, d_in: int, d_out: int, r: int) -> int:
    return 2 * n * r * (d_in + d_out)


def saved_activation_elems(wl: "Workload", mode: str) -> int:
    """Elements the layer path keeps from the forward for the backward: Z and
    H (n r each) per layer under CoLA, Z alone under CoLA-M, nothing for
    inference.  For a block with one rank r that is App. C's low-rank terms:
    +14nr for CoLA, 7nr for CoLA-M (whose 2nd of block inputs lies outside
    the layers)."""
    per = {"cola": 2, "cola_m": 1, "infer": 0}[mode]
    return sum(per * wl.n * l.r for l in wl.layers)


def llama_block(d: int, d_ff: int, r: int) -> tuple:
    return (
        Layer("q", d, d, r, "x_attn"),
        Layer("k", d, d, r, "x_attn"),
        Layer("v", d, d, r, "x_attn"),
        Layer("o", d, d, r, "x_o"),
        Layer("gate", d, d_ff, r, "x_mlp"),
        Layer("up", d, d_ff, r, "x_mlp"),
        Layer("down", d_ff, d, r, "x_down"),
    )


def paper_flops_full_rank(n: int, d: int, d_ff: int) -> float:
    """Table 3, full-rank row: 24nd^2 + 12n^2d + 18ndd_ff."""
    return 24 * n * d * d + 12 * n * n * d + 18 * n * d * d_ff


def paper_flops_cola(n: int, d: int, d_ff: int, r: int) -> float:
    """Table 3, CoLA row: 48ndr + 12n^2d + 18nr(d + d_ff)."""
    return 48 * n * d * r + 12 * n * n * d + 18 * n * r * (d + d_ff)


WORKLOADS = {
    "60m-q": Workload("60m-q", 2048, (Layer("q", 512, 512, 128, "x_attn"),), fused_qkv=False,
                      desc="single CoLA layer, LLaMA-60M q-proj shape, n=2048, 512->512, r=128",
                      seqs=8),
    "60m": Workload("60m", 65536, llama_block(512, 1376, 128),
                    desc="LLaMA-60M-shaped CoLA block, 7 layers, d=512, d_ff=1376, r=128, "
                         "65536 tokens (256 x 256)", seqs=256),
    "350m": Workload("350m", 131072, llama_block(1024, 2736, 256),
                     desc="LLaMA-350M-shaped CoLA block, d=1024, d_ff=2736, r=256, 131072 tokens "
                          "(512 x 256), fused QKV A-GEMM (N=768)", seqs=512),
    "1b": Workload("1b", 65536, llama_block(2048, 5461, 512), modes=("cola", "cola_m"),
                   desc="LLaMA-1B-shaped CoLA block, d=2048, d_ff=5461, r=512, 65536 tokens "
                        "(256 x 256), fused QKV A-GEMM (N=1536)", seqs=256),
    "7b": Workload("7b", 32768, llama_block(4096, 11008, 1024), modes=("cola_m", "cola"),
                   desc="LLaMA-7B-shaped CoLA block, d=4096, d_ff=11008, r=1024, 32768 tokens "
                        "(128 x 256)", seqs=128),
    # the 7B block at a quarter of its tokens: small enough for ncu captures
    # with many metrics, large enough that every GEMM keeps its tile
    # configuration (CTA pairs)
    "7b-8k": Workload("7b-8k", 8192, llama_block(4096, 11008, 1024), modes=("cola_m", "cola"),
                      desc="LLaMA-7B-shaped CoLA block, 8192 tokens (32 x 256), for profiling", seqs=32),
    "1b-o": Workload("1b-o", 65536, (Layer("o", 2048, 2048, 512, "x_o"),), fused_qkv=False,
                     desc="single CoLA layer, LLaMA-1B o-proj shape, 65536 tokens, 2048->2048, r=512", seqs=256),
    # the same blocks with the gated MLP chained through the library
    "60m-gated": Workload("60m-gated", 65536, llama_block(512, 1376, 128), gated=True,
                          desc="LLaMA-60M-shaped CoLA block with the gated MLP (M = Y_gate * Y_up fused), "
                               "65536 tokens", seqs=256),
    "1b-gated": Workload("1b-gated", 65536, llama_block(2048, 5461, 512), modes=("cola", "cola_m"), gated=True,
                         desc="LLaMA-1B-shaped CoLA block with the gated MLP (M = Y_gate * Y_up fused), "
                              "65536 tokens", seqs=256),
    "7b-gated": Workload("7b-gated", 32768, llama_block(4096, 11008, 1024), modes=("cola_m", "cola"), gated=True,
                         desc="LLaMA-7B-shaped CoLA block with the gated MLP (M = Y_gate * Y_up fused), "
                              "32768 tokens", seqs=128),
    # inference at the pre-training shapes with 32 sequences of 256 tokens (App. E.2)
    "1b-infer": Workload("1b-infer", 8192, llama_block(2048, 5461, 512), modes=("infer",), phase="infer", desc="LLaMA-1B-shaped CoLA block, forward only (inference), d=2048, "
                                          "d_ff=5461, r=512, 8192 tokens (32 x 256)", seqs=32),
    "7b-infer": Workload("7b-infer", 8192, llama_block(4096, 11008, 1024), modes=("infer",), phase="infer", desc="LLaMA-7B-shaped CoLA block, forward only (inference), d=4096, "
                                          "d_ff=11008, r=1024, 8192 tokens (32 x 256)", seqs=32),
    "1b-infer-gated": Workload("1b-infer-gated", 8192, llama_block(2048, 5461, 512), modes=("infer",),
                               phase="infer", gated=True,
                               desc="LLaMA-1B-shaped CoLA block with the gated MLP, forward only (inference), "
                                    "8192 tokens (32 x 256)", seqs=32),
    "7b-infer-gated": Workload("7b-infer-gated", 8192, llama_block(4096, 11008, 1024), modes=("infer",),
                               phase="infer", gated=True,
                               desc="LLaMA-7B-shaped CoLA block with the gated MLP, forward only (inference), "
                                    "8192 tokens (32 x 256)", seqs=32),
    # one new token for each of 32 sequences: every GEMM has a few output tiles
    # (split over K across the SMs) and streams its weights
    "1b-decode": Workload("1b-decode", 32, llama_block(2048, 5461, 512), modes=("infer",), phase="infer", desc="LLaMA-1B-shaped CoLA block, forward only, 32 tokens (one per sequence)",
                          seqs=32, seq_len=1),
    "7b-decode": Workload("7b-decode", 32, llama_block(4096, 11008, 1024), modes=("infer",), phase="infer", desc="LLaMA-7B-shaped CoLA block, forward only, 32 tokens (one per sequence)",
                          seqs=32, seq_len=1),
}
