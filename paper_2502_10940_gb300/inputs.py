"""Seeded synthetic inputs for the CoLA layer -- shared by the CUDA path's
tests/bench and by the oracle's tests.

This module draws random numbers and lays them out; it holds none of the
layer's arithmetic.  Distributions: activations X and upstream gradients dY
~ N(0, 1); factors A ~ N(0, 1/d_in) and B ~ N(0, 1/r) (zero-mean Gaussian
with variance 1/fan_in), all rounded once to bf16 (round to nearest even).
The paper trains on C4 (Sec. 5.1); no dataset is used here -- these
Gaussian stand-ins only give the shapes and value scales of that workload.

A tensor whose logical width is not a multiple of 8 elements gets a padded
row pitch (``ld``) so that every row starts 16-byte aligned; the padding
columns are filled with ``pad_value`` (a large value by default, so that any
read of the padding shows up in a result).
"""
from __future__ import annotations

import torch

PAD_VALUE = 4096.0

# stable per-tensor sub-streams of one base seed
_STREAM = {"X": 1, "A": 2, "B": 3, "dY": 4}


def padded_ld(cols: int, align_elems: int = 8) -> int:
    return (cols + align_elems - 1) // align_elems * align_elems


def normal_bf16(rows: int, cols: int, std: float, seed: int, device="cpu", ld: int | None = None,
                pad_value: float = PAD_VALUE) -> torch.Tensor:
    """[rows x cols] bf16 view with row pitch ``ld`` (>= cols), N(0, std^2)."""
    ld = cols if ld is None else ld
    assert ld >= cols
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    buf = torch.empty((rows, ld), dtype=torch.bfloat16, device=device)
    if ld > cols:
        buf[:, cols:].fill_(pad_value)
    v = torch.randn((rows, cols), generator=g, device=device, dtype=torch.float32)
    if std != 1.0:
        v.mul_(std)
    buf[:, :cols].copy_(v)
    return buf[:, :cols]


def _sub(seed: int, name: str, layer: int = 0) -> int:
    return (int(seed) * 1000003 + layer * 101 + _STREAM[name]) & 0x7FFFFFFFFFFF


def layer_inputs(n: int, d_in: int, d_out: int, r: int, seed: int = 0, device="cpu",
                 layer: int = 0, with_x: bool = True, with_dy: bool = True):
    """X [n x d_in], A [r x d_in], B [d_out x r], dY [n x d_out] (bf16)."""
    out = {}
    if with_x:
        out["X"] = normal_bf16(n, d_in, 1.0, _sub(seed, "X", layer), device, ld=padded_ld(d_in))
    out["A"] = normal_bf16(r, d_in, d_in ** -0.5, _sub(seed, "A", layer), device, ld=padded_ld(d_in))
    out["B"] = normal_bf16(d_out, r, r ** -0.5, _sub(seed, "B", layer), device)
    if with_dy:
        out["dY"] = normal_bf16(n, d_out, 1.0, _sub(seed, "dY", layer), device, ld=padded_ld(d_out))
    return out


def activation(n: int, d: int, seed: int, device="cpu", layer: int = 0) -> torch.Tensor:
    """A shared layer input X [n x d] (e.g. the one X that q, k and v read)."""
    return normal_bf16(n, d, 1.0, _sub(seed, "X", layer), device, ld=padded_ld(d))


def bf16_bits(t: torch.Tensor):
    """Host numpy uint16 view of a bf16 tensor's bit patterns (logical columns
    only; copies to host if needed)."""
    t = t.detach()
    if t.device.type != "cpu":
        t = t.cpu()
    return t.contiguous().view(torch.int16).numpy().view("uint16")
