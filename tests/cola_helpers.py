"""Shared pieces of the GPU parity tests: run the layer through the C ABI,
run the oracle on the same inputs, compare with the stated tolerance.

Tolerance (bf16 outputs from bf16 inputs, fp32 accumulation), per tensor:
    ||g - o||_F / ||o||_F <= 5e-3   and   max|g - o| <= 3e-2 * max|o|
where o is the fp64 oracle on the exact same bf16 inputs.
"""
import numpy as np
import torch

import oracle
from paper_2502_10940_gb300 import cola
from paper_2502_10940_gb300 import inputs as I

REL_F = 5e-3
REL_MAX = 3e-2
SENTINEL = float("nan")


def padded_empty(rows, cols, ld, dtype=torch.bfloat16, device="cuda", fill=SENTINEL):
    buf = torch.full((rows, ld), fill, dtype=dtype, device=device)
    return buf[:, :cols]


def assert_close(name, got, ref, rel_f=REL_F, rel_max=REL_MAX):
    g = np.asarray(got, dtype=np.float64)
    o = np.asarray(ref, dtype=np.float64)
    assert g.shape == o.shape, (name, g.shape, o.shape)
    assert np.all(np.isfinite(g)), f"{name}: non-finite values"
    err_f = np.linalg.norm(g - o) / max(np.linalg.norm(o), 1e-300)
    err_m = np.abs(g - o).max() / max(np.abs(o).max(), 1e-300)
    assert err_f <= rel_f and err_m <= rel_max, f"{name}: rel_F={err_f:.3e} rel_max={err_m:.3e}"
    return err_f, err_m


def to64(t):
    return t.detach().float().cpu().double().numpy()


def padding_intact(full_buf_view, cols):
    """True if the columns beyond `cols` of a padded view still hold the sentinel."""
    base = full_buf_view
    ld = base.stride(0)
    if ld == cols:
        return True
    raw = torch.as_strided(base, (base.shape[0], ld), (ld, 1))
    return bool(torch.isnan(raw[:, cols:].float()).all())


def gpu_layer(inp, sigma="silu", mode="cola", wgrad_fp32=False, dA0=None, dB0=None):
    """fwd + bwd of one layer through cola_fwd / cola_bwd on cuda tensors."""
    X, A, B, dY = inp["X"], inp["A"], inp["B"], inp["dY"]
    n, d_in = X.shape
    r = A.shape[0]
    d_out = B.shape[0]
    d = cola.desc(n, d_in, d_out, r, ld_x=cola.ld_of(X), ld_y=cola.ld_of(dY), ld_a=cola.ld_of(A),
                  sigma=sigma, mode=mode, wgrad_fp32=wgrad_fp32)
    Y = padded_empty(n, d_out, cola.ld_of(dY))
    Z = torch.empty((n, r), dtype=torch.bfloat16, device="cuda")
    H = torch.empty((n, r), dtype=torch.bfloat16, device="cuda") if mode == "cola" else None
    ws = cola.workspace(d)
    cola.cola_fwd(d, X, A, B, Y, Z, H, ws)
    dX = padded_empty(n, d_in, cola.ld_of(X))
    if wgrad_fp32:
        dA = padded_empty(r, d_in, cola.ld_of(A), torch.float32)
        dA.copy_(dA0)
        dB = dB0.clone()
    else:
        dA = padded_empty(r, d_in, cola.ld_of(A))
        dB = torch.empty((d_out, r), dtype=torch.bfloat16, device="cuda")
    cola.cola_bwd(d, X, A, B, dY, Z, H, dX, dA, dB, ws)
    st, code = cola.cola_check_status(ws)
    assert st == 0, (st, code)
    return dict(Y=Y, Z=Z, H=H, dX=dX, dA=dA, dB=dB)


def oracle_layer(inp, sigma="silu", mode="cola", round_store=False):
    X, A, B, dY = (to64(inp[k]) for k in ("X", "A", "B", "dY"))
    Z, H, Y = oracle.fwd(X, A, B, sigma, round_store)
    dX, dA, dB, dZ = oracle.bwd(X, A, B, dY, Z, H if mode == "cola" else None, sigma, mode, round_store)
    return dict(Y=Y, Z=Z, H=H, dX=dX, dA=dA, dB=dB, dZ=dZ)


def make_inputs(n, d_in, d_out, r, seed=0, device="cuda"):
    """Generated on the CPU generator (cheap at test sizes), moved to the device
    with their padded pitch intact."""
    cpu = I.layer_inputs(n, d_in, d_out, r, seed=seed, device="cpu")
    out = {}
    for k, v in cpu.items():
        ld = v.stride(0)
        buf = torch.as_strided(v, (v.shape[0], ld), (ld, 1)).contiguous().to(device)
        out[k] = buf[:, :v.shape[1]]
    return out
