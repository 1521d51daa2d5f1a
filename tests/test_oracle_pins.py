"""Pins of the fp64 CPU oracle against what the paper and the mathematics fix.

Each test ties the oracle to something other than itself: a closed form, an
invariant the paper states, a limit from one of its proofs, central finite
differences, or an independent library routine.  A dropped term, a wrong
sign, a wrong index or a transposed operand anywhere in the oracle fails at
least one of them.
"""
import math

import numpy as np
import pytest

import oracle

RNG = np.random.default_rng(20250215)
SIGMAS = ["identity", "silu", "gelu"]


def _rand_layer(n, d_in, d_out, r, rng=RNG):
    X = rng.standard_normal((n, d_in))
    A = rng.standard_normal((r, d_in)) / math.sqrt(d_in)
    B = rng.standard_normal((d_out, r)) / math.sqrt(r)
    dY = rng.standard_normal((n, d_out))
    return X, A, B, dY


# --- sigma: closed forms and derivative identities -------------------------

def test_silu_closed_forms():
    # SiLU(z) = z / (1 + e^{-z}); at z = ln 3 the logistic factor is exactly 3/4.
    l3 = math.log(3.0)
    got = oracle.sigma("silu", np.array([0.0, l3, -l3, 1.0, 30.0, -800.0]))
    want = [0.0, 0.75 * l3, -0.25 * l3, math.e / (1.0 + math.e), 30.0 - 30.0 * math.exp(-30.0), 0.0]
    np.testing.assert_allclose(got, want, rtol=1e-14, atol=1e-300)
    # Props. 3.1/3.2 need sigma(0) = 0, sigma'(0) != 0, sigma''(0) != 0; for SiLU
    # sigma'(0) = 1/2 and sigma''(0) = 1/2.
    assert oracle.dsigma("silu", np.array([0.0]))[0] == 0.5
    h = 1e-4
    d2 = (oracle.dsigma("silu", np.array([h]))[0] - oracle.dsigma("silu", np.array([-h]))[0]) / (2 * h)
    assert abs(d2 - 0.5) < 1e-7


def test_gelu_matches_normal_cdf():
    special = pytest.importorskip("scipy.special")
    z = np.linspace(-7, 7, 141)
    np.testing.assert_allclose(oracle.sigma("gelu", z), z * special.ndtr(z), rtol=1e-13, atol=1e-300)
    assert oracle.sigma("gelu", np.array([1.0]))[0] == pytest.approx(0.8413447460685429, rel=1e-15)
    assert oracle.dsigma("gelu", np.array([0.0]))[0] == 0.5


@pytest.mark.parametrize("kind", SIGMAS)
def test_dsigma_is_derivative_of_sigma(kind):
    z = np.linspace(-9, 9, 181) + 0.0123
    h = 1e-6
    fd = (oracle.sigma(kind, z + h) - oracle.sigma(kind, z - h)) / (2 * h)
    np.testing.assert_allclose(oracle.dsigma(kind, z), fd, rtol=1e-7, atol=1e-9)


def test_identity_sigma():
    z = RNG.standard_normal(50)
    assert np.array_equal(oracle.sigma("identity", z), z)
    assert np.all(oracle.dsigma("identity", z) == 1.0)


# --- bf16 rounding used by round_store --------------------------------------

def test_round_bf16_ties_and_grid():
    u = 2.0 ** -8   # half the bf16 spacing at 1
    cases = {
        1.0 + u: 1.0,                      # tie -> even (1.0)
        1.0 + 3 * u: 1.0 + 4 * u,          # tie -> even (1 + 2^-6)
        1.0 + u + 2.0 ** -30: 1.0 + 2 * u,  # just above the tie rounds up
        -(1.0 + u): -1.0,
        3.0: 3.0,
        2.0 ** -130: 2.0 ** -130,           # bf16 subnormal, exact
        3 * 2.0 ** -134: 2.0 ** -132,       # subnormal tie -> even
        255.5: 256.0,                       # 8 significant bits: 255.5 is a tie -> 256
        254.5: 254.0,
    }
    x = np.array(list(cases.keys()))
    np.testing.assert_array_equal(oracle.round_bf16(x), np.array(list(cases.values())))


def test_round_bf16_matches_torch_on_float32_values():
    torch = pytest.importorskip("torch")
    v = (RNG.standard_normal(20000) * np.exp(RNG.uniform(-20, 20, 20000))).astype(np.float32)
    want = torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(oracle.round_bf16(v.astype(np.float64)), want)


# --- forward: Eq. (main-fwd) ----------------------------------------------------

def test_identity_sigma_reduces_to_BAX():
    # Sec. 3.3: with sigma = identity the layer is the plain low-rank product BAX;
    # token-major: Y = X (BA)^T, with BA formed first by a library matmul.
    X, A, B, _ = _rand_layer(37, 29, 41, 6)
    _, _, Y = oracle.fwd(X, A, B, "identity")
    np.testing.assert_allclose(Y, X @ (B @ A).T, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_output_rank_at_most_r(kind):
    # Y = B sigma(AX) with B in R^{d_out x r}: rank(Y) <= r (Sec. 3.2).
    X, A, B, _ = _rand_layer(60, 24, 32, 5)
    _, _, Y = oracle.fwd(X, A, B, kind)
    s = np.linalg.svd(Y, compute_uv=False)
    assert s[4] > 1e-3 * s[0]
    assert s[5] < 1e-12 * s[0]


def test_forward_elementwise_definition_small():
    # Z is A x per token, H = sigma(Z), Y = B H: checked on a 2-token example
    # whose values are worked by hand.
    X = np.array([[1.0, 2.0, 0.0], [0.0, -1.0, 3.0]])
    A = np.array([[1.0, 0.0, 1.0], [0.5, 0.5, 0.0]])
    B = np.array([[1.0, 0.0], [2.0, -1.0]])
    Z, H, Y = oracle.fwd(X, A, B, "identity")
    np.testing.assert_array_equal(Z, [[1.0, 1.5], [3.0, -0.5]])
    np.testing.assert_array_equal(Y, [[1.0, 0.5], [3.0, 6.5]])


def test_tau_limit_of_prop_3_1():
    # Proof of Prop. 3.1: A_tau = tau A*, B_tau = B* / (sigma'(0) tau) gives
    # B_tau sigma(A_tau X) -> B*A*X with an O(tau) error when sigma''(0) != 0.
    X, A, B, _ = _rand_layer(30, 12, 10, 4)
    _, _, Ylin = oracle.fwd(X, A, B, "identity")
    errs = []
    for tau in (1e-2, 5e-3, 2.5e-3):
        _, _, Yt = oracle.fwd(X, tau * A, B / (0.5 * tau), "silu")
        errs.append(np.linalg.norm(Yt - Ylin))
    assert errs[0] / errs[1] == pytest.approx(2.0, rel=0.02)
    assert errs[1] / errs[2] == pytest.approx(2.0, rel=0.02)


@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_lemma_rank_one_construction(kind):
    # Lemma (App. H, auxiliary lemmas): every row of A equal to u^T and B = [w, 0, ..., 0]
    # give B sigma(A X) = w sigma(u^T X) exactly.  In the backward only the
    # first column of dH is nonzero, so dA rows 1..r-1 vanish, and all
    # columns of H (hence of dB) coincide.
    n, d_in, d_out, r = 23, 9, 7, 4
    X, _, _, dY = _rand_layer(n, d_in, d_out, r)
    u = RNG.standard_normal(d_in)
    w = RNG.standard_normal(d_out)
    A = np.tile(u, (r, 1))
    B = np.zeros((d_out, r))
    B[:, 0] = w
    Z, H, Y = oracle.fwd(X, A, B, kind)
    v = oracle.sigma(kind, X @ u)
    np.testing.assert_allclose(Y, np.outer(v, w), rtol=1e-12, atol=1e-14)
    dX, dA, dB, dZ = oracle.bwd(X, A, B, dY, Z, H, kind, "cola")
    assert np.all(dA[1:] == 0.0)
    assert np.all(dZ[:, 1:] == 0.0)
    for j in range(1, r):
        assert np.array_equal(dB[:, j], dB[:, 0])
    assert np.abs(dA[0]).max() > 0


# --- backward: Sec. 3.4 ----------------------------------------------------------

def _loss(X, A, B, dY, kind):
    return float(np.sum(dY * oracle.fwd(X, A, B, kind)[2]))


def _fd_grad(f, P, h=1e-5):
    g = np.zeros_like(P)
    it = np.nditer(P, flags=["multi_index"])
    for _ in it:
        idx = it.multi_index
        old = P[idx]
        P[idx] = old + h
        fp = f()
        P[idx] = old - h
        fm = f()
        P[idx] = old
        g[idx] = (fp - fm) / (2 * h)
    return g


def _rel(a, b):
    return np.linalg.norm(a - b) / np.linalg.norm(b)


@pytest.mark.parametrize("kind", SIGMAS)
@pytest.mark.parametrize("mode", ["cola", "cola_m"])
def test_backward_matches_central_differences(kind, mode):
    # d = 8, r = 2, n = 5: the gradients of L = sum(dY * Y) w.r.t. X, A, B.
    n, d, r = 5, 8, 2
    X, A, B, dY = _rand_layer(n, d, d, r)
    Z, H, _ = oracle.fwd(X, A, B, kind)
    dX, dA, dB, _ = oracle.bwd(X, A, B, dY, Z, H if mode == "cola" else None, kind, mode)
    f = lambda: _loss(X, A, B, dY, kind)  # noqa: E731
    assert _rel(dX, _fd_grad(f, X)) < 1e-6
    assert _rel(dA, _fd_grad(f, A)) < 1e-6
    assert _rel(dB, _fd_grad(f, B)) < 1e-6


def test_backward_rectangular_central_differences():
    n, d_in, d_out, r = 4, 6, 9, 3
    X, A, B, dY = _rand_layer(n, d_in, d_out, r)
    Z, H, _ = oracle.fwd(X, A, B, "silu")
    dX, dA, dB, dZ = oracle.bwd(X, A, B, dY, Z, H, "silu", "cola")
    f = lambda: _loss(X, A, B, dY, "silu")  # noqa: E731
    assert _rel(dX, _fd_grad(f, X)) < 1e-6
    assert _rel(dA, _fd_grad(f, A)) < 1e-6
    assert _rel(dB, _fd_grad(f, B)) < 1e-6
    # dZ is the gradient of L at Z: perturb Z through an identity layer on top of H.
    g = np.zeros_like(Z)
    for t in range(n):
        for i in range(r):
            for s in (+1, -1):
                Zp = Z.copy()
                Zp[t, i] += s * 1e-5
                g[t, i] += s * np.sum(dY * (oracle.sigma("silu", Zp) @ B.T)) / 2e-5
    assert _rel(dZ, g) < 1e-6


@pytest.mark.parametrize("round_store", [False, True])
def test_cola_and_cola_m_gradients_identical(round_store):
    # CoLA saves Z and sigma(Z); CoLA-M saves Z and recomputes sigma(Z)
    # (Sec. 4.2): the gradients must be identical.
    X, A, B, dY = _rand_layer(33, 20, 28, 8)
    Z, H, _ = oracle.fwd(X, A, B, "silu", round_store)
    g1 = oracle.bwd(X, A, B, dY, Z, H, "silu", "cola", round_store)
    g2 = oracle.bwd(X, A, B, dY, Z, None, "silu", "cola_m", round_store)
    for a, b in zip(g1, g2):
        assert np.array_equal(a, b)


def test_qkv_fused_backward_central_differences():
    # q, k, v read one X (Fig. 4): dX is the sum of the three input gradients.
    n, d, r = 4, 8, 2
    X = RNG.standard_normal((n, d))
    As = [RNG.standard_normal((r, d)) / math.sqrt(d) for _ in range(3)]
    Bs = [RNG.standard_normal((d, r)) / math.sqrt(r) for _ in range(3)]
    dYs = [RNG.standard_normal((n, d)) for _ in range(3)]
    Zs, Hs, _ = oracle.fwd_qkv(X, As, Bs, "silu")
    dX, dAs, dBs, _ = oracle.bwd_qkv(X, As, Bs, dYs, Zs, Hs, "silu", "cola")

    def f():
        return sum(float(np.sum(dY * oracle.fwd(X, A, B, "silu")[2])) for A, B, dY in zip(As, Bs, dYs))

    assert _rel(dX, _fd_grad(f, X)) < 1e-6
    for j in range(3):
        assert _rel(dAs[j], _fd_grad(f, As[j])) < 1e-6
        assert _rel(dBs[j], _fd_grad(f, Bs[j])) < 1e-6


@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_backward_matches_torch_autograd_fp64(kind):
    torch = pytest.importorskip("torch")
    n, d_in, d_out, r = 37, 24, 40, 8
    X, A, B, dY = _rand_layer(n, d_in, d_out, r)
    Xt, At, Bt = (torch.tensor(v, requires_grad=True) for v in (X, A, B))
    act = torch.nn.functional.silu if kind == "silu" else (lambda z: torch.nn.functional.gelu(z))
    Yt = act(Xt @ At.T) @ Bt.T
    Yt.backward(torch.tensor(dY))
    Z, H, Y = oracle.fwd(X, A, B, kind)
    dX, dA, dB, _ = oracle.bwd(X, A, B, dY, Z, H, kind, "cola")
    np.testing.assert_allclose(Y, Yt.detach().numpy(), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(dX, Xt.grad.numpy(), rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(dA, At.grad.numpy(), rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(dB, Bt.grad.numpy(), rtol=1e-10, atol=1e-11)


def test_round_store_places_rounding_at_storage_points():
    # round_store: Z and H on the bf16 grid, H = bf16(sigma(bf16(Z))).
    X, A, B, dY = _rand_layer(12, 16, 8, 4)
    Z, H, Y = oracle.fwd(X, A, B, "silu", round_store=True)
    Z0, _, _ = oracle.fwd(X, A, B, "silu")
    np.testing.assert_array_equal(Z, oracle.round_bf16(Z0))
    np.testing.assert_array_equal(H, oracle.round_bf16(oracle.sigma("silu", Z)))
    _, _, _, dZ = oracle.bwd(X, A, B, dY, Z, H, "silu", "cola", round_store=True)
    np.testing.assert_array_equal(dZ, oracle.round_bf16(dZ))


# --- sampled routines equal the full ones -------------------------------------

def _bf16_valued(shape, std=1.0):
    v = (RNG.standard_normal(shape) * std).astype(np.float32)
    bits = (v.view(np.uint32) >> 16).astype(np.uint16)   # truncation: any bf16 grid point will do
    return bits, oracle.widen_bf16(bits)


@pytest.mark.parametrize("round_store", [False, True])
def test_sampled_oracle_equals_full(round_store):
    n, d_in, d_out, r = 50, 40, 24, 8
    Xb, X = _bf16_valued((n, d_in))
    Ab, A = _bf16_valued((r, d_in), d_in ** -0.5)
    Bb, B = _bf16_valued((d_out, r), r ** -0.5)
    dYb, dY = _bf16_valued((n, d_out))
    Z, H, Y = oracle.fwd(X, A, B, "silu", round_store)
    dX, dA, dB, dZ = oracle.bwd(X, A, B, dY, Z, H, "silu", "cola", round_store)
    rows = np.array([0, 7, 49, 13])
    z, h, y, dz, dx = oracle.rows_bf16(Xb, Ab, Bb, rows, dYb, "silu", round_store)
    for got, full in ((z, Z), (h, H), (y, Y), (dz, dZ), (dx, dX)):
        np.testing.assert_allclose(got, full[rows], rtol=1e-13, atol=1e-15)
    ii, kk = np.array([0, 3, 7, 7]), np.array([1, 39, 0, 20])
    np.testing.assert_allclose(oracle.dA_entries_bf16(Xb, Ab, Bb, dYb, ii, kk, "silu", round_store),
                               dA[ii, kk], rtol=1e-13, atol=1e-15)
    oo, ii2 = np.array([0, 23, 5]), np.array([7, 0, 4])
    np.testing.assert_allclose(oracle.dB_entries_bf16(Xb, Ab, dYb, oo, ii2, "silu", round_store),
                               dB[oo, ii2], rtol=1e-13, atol=1e-15)


def test_sampled_oracle_padded_row_pitch():
    # X and dY with a padded row pitch (ld > logical width): the padding is never read.
    n, d_in, d_out, r = 20, 13, 11, 4
    Xb, X = _bf16_valued((n, d_in))
    Ab, A = _bf16_valued((r, d_in), 0.3)
    Bb, B = _bf16_valued((d_out, r), 0.5)
    dYb, dY = _bf16_valued((n, d_out))
    Xp = np.full((n, 16), 0x7FC0, dtype=np.uint16)   # NaN padding
    Xp[:, :d_in] = Xb
    dYp = np.full((n, 16), 0x7FC0, dtype=np.uint16)
    dYp[:, :d_out] = dYb
    Z, H, Y = oracle.fwd(X, A, B, "silu")
    dX, dA, dB, dZ = oracle.bwd(X, A, B, dY, Z, H, "silu", "cola")
    rows = np.arange(n)
    z, h, y, dz, dx = oracle.rows_bf16(Xp, Ab, Bb, rows, dYp, "silu", d_in=d_in, d_out=d_out)
    np.testing.assert_allclose(y, Y, rtol=1e-13)
    np.testing.assert_allclose(dx, dX, rtol=1e-13)
    ii, kk = np.array([1, 3]), np.array([12, 0])
    np.testing.assert_allclose(oracle.dA_entries_bf16(Xp, Ab, Bb, dYp, ii, kk, "silu", d_out=d_out),
                               dA[ii, kk], rtol=1e-13)
    oo, ii2 = np.array([10, 0]), np.array([3, 2])
    np.testing.assert_allclose(oracle.dB_entries_bf16(Xp, Ab, dYp, oo, ii2, "silu"), dB[oo, ii2], rtol=1e-13)


# --- CoLA-M block-level recompute of the up-projection (Sec. 4.2, App. C) ---

@pytest.mark.parametrize("kind", SIGMAS)
def test_recompute_up_reproduces_forward_output(kind):
    # recomputing B sigma(.) from the saved Z gives the forward's Y: the C
    # forward's loops against sigma + a numpy product
    X, A, B, _ = _rand_layer(23, 17, 31, 5)
    Z, _, Y = oracle.fwd(X, A, B, kind)
    np.testing.assert_allclose(oracle.recompute_up(Z, B, kind), Y, rtol=1e-12, atol=1e-12)


def test_recompute_up_worked_example():
    # one token, r = 2: Z = [0, 1], B = [[1, 2], [-3, 0.5]], SiLU:
    # sigma(0) = 0 and sigma(1) = 1 / (1 + e^-1), so Y = [2 s, 0.5 s] with s = sigma(1)
    s = 1.0 / (1.0 + math.exp(-1.0))
    Y = oracle.recompute_up(np.array([[0.0, 1.0]]), np.array([[1.0, 2.0], [-3.0, 0.5]]), "silu")
    np.testing.assert_allclose(Y, [[2.0 * s, 0.5 * s]], rtol=1e-15)


# --- gated MLP: M = Y_gate * Y_up (Fig. 4, Sec. 3.2, App. E) ---

def test_gate_up_closed_form_identity_sigma():
    # sigma = identity and every row of B_up the same vector b: Y_up[t, o] =
    # x_t . (A_up^T b) for every o, so M[t, o] = (X (B_g A_g)^T)[t, o] c_t with
    # c = X A_up^T b -- computed here with the factors multiplied first
    rng = np.random.default_rng(41)
    n, d_in, d_ff, r = 7, 12, 10, 3
    X = rng.standard_normal((n, d_in))
    Ag = rng.standard_normal((r, d_in))
    Bg = rng.standard_normal((d_ff, r))
    Au = rng.standard_normal((r, d_in))
    b = rng.standard_normal(r)
    Bu = np.tile(b, (d_ff, 1))
    *_, M = oracle.gated_fwd(X, Ag, Bg, Au, Bu, "identity")
    c = X @ (Au.T @ b)
    np.testing.assert_allclose(M, (X @ (Bg @ Ag).T) * c[:, None], rtol=1e-12, atol=1e-12)


def test_gate_up_product_worked_example():
    # two entries by hand: 2 x (-3) = -6 and 0.5 x 4 = 2; the backward swaps
    # the factors: dY_gate = dM * Y_up, dY_up = dM * Y_gate
    M = oracle.gate_up_product(np.array([[2.0, 0.5]]), np.array([[-3.0, 4.0]]))
    np.testing.assert_array_equal(M, [[-6.0, 2.0]])
    dYg, dYu = oracle.gate_up_backward(np.array([[1.0, -2.0]]), np.array([[2.0, 0.5]]), np.array([[-3.0, 4.0]]))
    np.testing.assert_array_equal(dYg, [[-3.0, -8.0]])
    np.testing.assert_array_equal(dYu, [[2.0, -1.0]])


@pytest.mark.parametrize("kind", ["silu", "gelu"])
def test_gated_mlp_central_differences(kind):
    # the whole gated MLP of one block: M = gate(X) * up(X), out = down(M);
    # L = sum(dOut * out).  Its gradients through the oracle's pieces (down
    # backward -> dM -> product backward -> the two layers' backward, dX
    # summed) against central differences of L w.r.t. X, A_gate, B_up, A_down
    rng = np.random.default_rng(43)
    n, d, d_ff, r = 4, 6, 8, 2
    X = rng.standard_normal((n, d))
    Ag, Au = (rng.standard_normal((r, d)) / math.sqrt(d) for _ in range(2))
    Bg, Bu = (rng.standard_normal((d_ff, r)) / math.sqrt(r) for _ in range(2))
    Ad = rng.standard_normal((r, d_ff)) / math.sqrt(d_ff)
    Bd = rng.standard_normal((d, r)) / math.sqrt(r)
    dOut = rng.standard_normal((n, d))

    def loss():
        *_, M = oracle.gated_fwd(X, Ag, Bg, Au, Bu, kind)
        return float(np.sum(dOut * oracle.fwd(M, Ad, Bd, kind)[2]))

    Zg, Hg, Yg, Zu, Hu, Yu, M = oracle.gated_fwd(X, Ag, Bg, Au, Bu, kind)
    Zd, Hd, _ = oracle.fwd(M, Ad, Bd, kind)
    dM, dAd, _, _ = oracle.bwd(M, Ad, Bd, dOut, Zd, Hd, kind, "cola")
    dYg, dYu = oracle.gate_up_backward(dM, Yg, Yu)
    dXg, dAg, _, _ = oracle.bwd(X, Ag, Bg, dYg, Zg, Hg, kind, "cola")
    dXu, _, dBu, _ = oracle.bwd(X, Au, Bu, dYu, Zu, Hu, kind, "cola")
    assert _rel(dXg + dXu, _fd_grad(loss, X)) < 1e-6
    assert _rel(dAg, _fd_grad(loss, Ag)) < 1e-6
    assert _rel(dBu, _fd_grad(loss, Bu)) < 1e-6
    assert _rel(dAd, _fd_grad(loss, Ad)) < 1e-6
