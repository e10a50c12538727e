"""Pins for the fp64 oracle: checks against things other than the oracle itself.

Each test fixes one step of the oracle by a fact the paper or the mathematics
determines -- finite differences of the forward loss, an exact invariant, a
special case that reduces to a textbook routine, or a hand-derived closed
form -- chosen so that a dropped term, a wrong sign or index, or a transposed
operand in the oracle fails at least one of them.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ---------------------------------------------------------------------------
# Independent forward model: the loss the error signal is the gradient of.
# L(h) = s * sum_t CE(RMSNorm(h_t) W_U^T, y_t)   (Sec. 3.1, App. E)
# ---------------------------------------------------------------------------
def forward_loss(h, w, W_U, y, eps, s):
    rho = np.sqrt(np.mean(h * h, axis=1, keepdims=True) + eps)
    z = (h / rho * w) @ W_U.T
    m = z.max(axis=1, keepdims=True)
    lse = (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]
    return s * float(np.sum(lse - z[np.arange(len(y)), y]))


def fd_grad(f, x, step=1e-6):
    gr = np.zeros_like(x)
    it = np.nditer(x, flags=["multi_index"])
    for _ in it:
        i = it.multi_index
        old = x[i]
        x[i] = old + step
        fp = f(x)
        x[i] = old - step
        fm = f(x)
        x[i] = old
        gr[i] = (fp - fm) / (2 * step)
    return gr


def rel_err(a, b):
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def _toy(T=4, d=8, V=16, seed=0, scale_h=1.0):
    rng = np.random.default_rng(seed)
    h = rng.standard_normal((T, d)) * scale_h
    w = 1.0 + 0.1 * rng.standard_normal(d)
    W_U = 0.5 * rng.standard_normal((V, d))
    y = rng.integers(0, V, T).astype(np.int32)
    return h, w, W_U, y


def test_error_signal_matches_finite_differences():
    """g~ = dL/dh exactly when the clamp is inactive (Eq. gproj + Eq. rmsnorm-vjp)."""
    h, w, W_U, y = _toy()
    s = 1.0 / len(y)
    out = oracle.error_signal(h, w, W_U, y, eps=1e-6, min_rms=0.5, s=s)
    assert np.all(out["rho"] > 0.5)
    fd = fd_grad(lambda x: forward_loss(x, w, W_U, y, 1e-6, s), h.copy())
    assert rel_err(out["g_tilde"], fd) < 1e-7


def test_error_signal_loss_scale_is_linear():
    h, w, W_U, y = _toy(seed=3)
    a = oracle.error_signal(h, w, W_U, y, s=1.0)["g_tilde"]
    b = oracle.error_signal(h, w, W_U, y, s=0.25)["g_tilde"]
    assert rel_err(0.25 * a, b) < 1e-14


def test_pre_vjp_signal_is_gradient_wrt_unembedding_input():
    """Eq. (gproj): g = e W_U is the exact gradient w.r.t. the unembedding input yhat."""
    h, w, W_U, y = _toy(seed=1)
    out = oracle.error_signal(h, w, W_U, y, s=1.0)
    rho = np.sqrt(np.mean(h * h, axis=1, keepdims=True) + 1e-6)
    yhat = h / rho * w

    def loss_of_yhat(yh):
        z = yh @ W_U.T
        m = z.max(axis=1, keepdims=True)
        lse = (m + np.log(np.exp(z - m).sum(axis=1, keepdims=True)))[:, 0]
        return float(np.sum(lse - z[np.arange(len(y)), y]))

    fd = fd_grad(loss_of_yhat, yhat.copy())
    assert rel_err(out["g"], fd) < 1e-7


def test_min_rms_clamp_scales_only_the_prefactor():
    """A token with rho < rho_min: g~ = (rho / rho_min) * dL/dh (clamp on 1/rho only)."""
    h, w, W_U, y = _toy(T=3, seed=2)
    h[1] *= 0.2  # rho ~ 0.2 < 0.5
    out = oracle.error_signal(h, w, W_U, y, eps=1e-6, min_rms=0.5, s=1.0)
    assert out["rho"][1] < 0.5 and out["rho"][0] > 0.5 and out["rho"][2] > 0.5
    fd = fd_grad(lambda x: forward_loss(x, w, W_U, y, 1e-6, 1.0), h.copy())
    expect = fd.copy()
    expect[1] *= out["rho"][1] / 0.5
    assert rel_err(out["g_tilde"], expect) < 1e-7
    # and with the clamp floor at 0 the plain gradient comes back
    out0 = oracle.error_signal(h, w, W_U, y, eps=1e-6, min_rms=0.0, s=1.0)
    assert rel_err(out0["g_tilde"], fd) < 1e-7


def test_rows_of_error_sum_to_zero():
    """softmax(z) - 1_y sums to zero over the vocabulary for every token."""
    h, w, W_U, y = _toy(T=6, V=40, seed=4)
    out = oracle.error_signal(h, w, W_U, y, s=1.0, want_e=True)
    assert np.max(np.abs(out["e"].sum(axis=1))) < 1e-12
    assert np.all(out["e"][np.arange(6), y] < 0)


def test_confident_token_target_entry_closed_form():
    """Two-word vocabulary, logits (40, 0), target 0: p_1 = 1 / (1 + e^40) ~ 4.2e-18, so
    e_0 = -p_1, e_1 = p_1 and g = e W_U = -40 p_1 (Sec. 3.1 step 2), values that p_0 - 1
    cannot carry in fp64 (1 / (1 + 4.2e-18) rounds to 1)."""
    h, w = np.array([[1.0]]), np.array([1.0])  # eps = 0: rho = 1, yhat = 1
    W_U = np.array([[40.0], [0.0]])
    out = oracle.error_signal(h, w, W_U, np.array([0]), eps=0.0, min_rms=0.0, s=1.0, want_e=True)
    p1 = 1.0 / (1.0 + math.exp(40.0))
    assert abs(out["e"][0, 1] - p1) <= 1e-14 * p1
    assert abs(out["e"][0, 0] + p1) <= 1e-14 * p1
    assert abs(out["g"][0, 0] + 40.0 * p1) <= 1e-14 * 40.0 * p1


def test_eps0_vjp_orthogonal_to_h():
    """At eps = 0 the RMSNorm VJP is orthogonal to h, clamped tokens included."""
    h, w, W_U, y = _toy(T=5, seed=5)
    h[2] *= 0.1
    out = oracle.error_signal(h, w, W_U, y, eps=0.0, min_rms=0.5, s=1.0)
    for t in range(5):
        gt = out["g_tilde"][t]
        assert abs(gt @ h[t]) <= 1e-12 * np.linalg.norm(gt) * np.linalg.norm(h[t])


def test_vocab_of_one_gives_zero_signal():
    h, w, W_U, y = _toy(V=1, seed=6)
    y[:] = 0
    out = oracle.error_signal(h, w, W_U, y, s=1.0, want_e=True)
    assert np.all(out["e"] == 0.0)
    assert np.all(out["g_tilde"] == 0.0)
    A = np.random.default_rng(0).standard_normal((len(y), 5))
    assert np.all(oracle.pseudograd(out["g_tilde"], A) == 0.0)


def test_equal_unembedding_rows_give_zero_signal():
    h, w, W_U, y = _toy(V=12, seed=7)
    W_U[:] = W_U[0]
    out = oracle.error_signal(h, w, W_U, y, s=1.0)
    assert np.max(np.abs(out["g"])) < 1e-14
    assert np.max(np.abs(out["g_tilde"])) < 1e-13


def test_logsumexp_and_mean_ce_against_library():
    scipy_special = pytest.importorskip("scipy.special")
    h, w, W_U, y = _toy(T=7, V=33, seed=8)
    out = oracle.error_signal(h, w, W_U, y, eps=1e-6, s=1.0)
    rho = np.sqrt(np.mean(h * h, axis=1) + 1e-6)
    z = (h / rho[:, None] * w) @ W_U.T
    assert np.allclose(out["lse"], scipy_special.logsumexp(z, axis=1), rtol=0, atol=1e-13)
    assert np.allclose(out["zy"], z[np.arange(7), y], rtol=0, atol=1e-13)
    assert np.allclose(out["rho"], rho, rtol=1e-15, atol=0)
    ce = oracle.mean_ce(out["lse"], out["zy"])
    assert abs(ce - forward_loss(h, w, W_U, y, 1e-6, 1.0 / 7)) < 1e-13


def test_row_subset_equals_full():
    h, w, W_U, y = _toy(T=9, seed=9)
    full = oracle.error_signal(h, w, W_U, y, s=0.5)
    rows = [7, 0, 3]
    sub = oracle.error_signal(h, w, W_U, y, s=0.5, rows=rows)
    for k in ("rho", "lse", "zy"):
        assert np.array_equal(sub[k], full[k][rows])
    assert np.array_equal(sub["g_tilde"], full["g_tilde"][rows])


def test_pseudograd_against_matmul_and_pairs():
    rng = np.random.default_rng(10)
    g = rng.standard_normal((13, 6))
    A = rng.standard_normal((13, 9))
    G = oracle.pseudograd(g, A)
    assert G.shape == (6, 9)
    assert np.allclose(G, g.T @ A, rtol=1e-13, atol=1e-13)
    ii = np.array([0, 5, 2, 5])
    jj = np.array([8, 0, 4, 8])
    Gs = oracle.pseudograd(g, A, pairs=(ii, jj))
    assert np.array_equal(Gs, G[ii, jj])


def test_identity_above_layer_invariant():
    """With nothing above layer l (h = h0 + A W^T, the MLP output added to the
    residual and fed straight to the final norm), the pseudogradient is the
    exact down-projection gradient: dL/dW = g~(h)^T A (Sec. 2.1, Eq. decomp with R = 0)."""
    rng = np.random.default_rng(11)
    T, d, d_ff, V = 5, 6, 7, 10
    h0 = rng.standard_normal((T, d))
    A = rng.standard_normal((T, d_ff))
    W = 0.1 * rng.standard_normal((d, d_ff))
    w = 1.0 + 0.1 * rng.standard_normal(d)
    W_U = 0.5 * rng.standard_normal((V, d))
    y = rng.integers(0, V, T).astype(np.int32)
    s = 1.0 / T
    h = h0 + A @ W.T
    out = oracle.error_signal(h, w, W_U, y, eps=1e-6, min_rms=0.5, s=s)
    assert np.all(out["rho"] > 0.5)
    G = oracle.pseudograd(out["g_tilde"], A)
    fd = fd_grad(lambda Wx: forward_loss(h0 + A @ Wx.T, w, W_U, y, 1e-6, s), W.copy())
    assert rel_err(G, fd) < 1e-7


def _ev(expr):
    return float(eval(expr, {"__builtins__": {}}, {"exp": math.exp, "log": math.log, "sqrt": math.sqrt}))


def test_hand_derived_closed_form():
    fx = json.load(open(os.path.join(GOLDEN, "closed_form_t1_d2_v2.json")))
    inp = fx["inputs"]
    w = np.array(inp["w"])
    W_U = np.array(inp["W_U"])
    y = np.array(inp["y"], dtype=np.int32)
    for name, case in fx["cases"].items():
        h = np.array(case["h"])
        out = oracle.error_signal(h, w, W_U, y, eps=inp["eps"], min_rms=inp["min_rms"], s=inp["s"])
        assert abs(out["rho"][0] - _ev(case["rho"])) < 1e-15, name
        assert abs(out["lse"][0] - _ev(case["lse"])) < 1e-15, name
        assert np.allclose(out["g"][0], [_ev(e) for e in case["g"]], rtol=0, atol=1e-15), name
        assert np.allclose(out["g_tilde"][0], [_ev(e) for e in case["g_tilde"]], rtol=0,
                           atol=1e-15), name
        if "G" in case:
            G = oracle.pseudograd(out["g_tilde"], np.array(inp["A"]))
            assert np.allclose(G, [[_ev(e) for e in r] for r in case["G"]], rtol=0, atol=1e-15)
            W_new, _ = oracle.sgd_update(np.array(inp["W"], dtype=np.float32), G, inp["lr"])
            expect = np.array([[_ev(e) for e in r] for r in case["W_new"]]).astype(np.float32)
            assert np.array_equal(W_new, expect)
        if "ce" in case:
            assert abs(oracle.mean_ce(out["lse"], out["zy"]) - _ev(case["ce"])) < 1e-15


def test_symbolic_gradient_exact():
    """Exact symbolic differentiation of the forward loss (sympy) on a 2x3x3 case."""
    sp = pytest.importorskip("sympy")
    rng = np.random.default_rng(12)
    T, d, V = 2, 3, 3
    hv = np.round(rng.standard_normal((T, d)), 3)
    wv = np.round(1 + 0.1 * rng.standard_normal(d), 3)
    Wv = np.round(rng.standard_normal((V, d)), 3)
    yv = np.array([2, 0], dtype=np.int32)
    eps = sp.Rational(1, 1000)
    H = sp.Matrix(T, d, lambda i, j: sp.Symbol(f"h{i}{j}"))
    L = 0
    for t in range(T):
        rho = sp.sqrt(sum(H[t, j] ** 2 for j in range(d)) / d + eps)
        z = [sum(sp.nsimplify(wv[j]) * H[t, j] / rho * sp.nsimplify(Wv[v, j]) for j in range(d))
             for v in range(V)]
        L += sp.log(sum(sp.exp(zv) for zv in z)) - z[int(yv[t])]
    subs = {H[i, j]: sp.nsimplify(hv[i, j]) for i in range(T) for j in range(d)}
    grad = np.array([[float(sp.diff(L, H[i, j]).evalf(30, subs=subs)) for j in range(d)]
                     for i in range(T)])
    out = oracle.error_signal(hv, wv, Wv, yv, eps=1e-3, min_rms=0.0, s=1.0)
    assert rel_err(out["g_tilde"], grad) < 1e-13


def test_bf16_input_upcast_is_exact():
    torch = pytest.importorskip("torch")
    x = torch.randn(257, dtype=torch.float32).to(torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(oracle.bf16_bits_to_f64(bits), x.to(torch.float64).numpy())
    # the oracle reads bf16 the same way: a bf16 run equals an fp64 run on the upcast values
    rng = np.random.default_rng(13)
    h = torch.tensor(rng.standard_normal((3, 16)), dtype=torch.bfloat16)
    w = torch.tensor(1 + 0.1 * rng.standard_normal(16), dtype=torch.bfloat16)
    W_U = torch.tensor(0.3 * rng.standard_normal((20, 16)), dtype=torch.bfloat16)
    y = np.array([1, 19, 4], dtype=np.int32)
    as_bits = lambda t: t.view(torch.int16).numpy().view(np.uint16)
    a = oracle.error_signal(as_bits(h), as_bits(w), as_bits(W_U), y, s=1.0)
    b = oracle.error_signal(h.double().numpy(), w.double().numpy(), W_U.double().numpy(), y, s=1.0)
    assert np.array_equal(a["g_tilde"], b["g_tilde"])


def test_sgd_update_exact_cases_and_bf16_rounding():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(14)
    W = (0.02 * rng.standard_normal(4096)).astype(np.float32)
    G = rng.standard_normal(4096)
    W0, b0 = oracle.sgd_update(W, G, 0.0)
    assert np.array_equal(W0, W)  # lr = 0 leaves the master bit-identical
    W1, b1 = oracle.sgd_update(W, G, 1e-3)
    assert np.array_equal(W1, (W.astype(np.float64) - 1e-3 * G).astype(np.float32))
    # round-to-nearest-even to bf16 agrees with torch's conversion bit for bit
    ref = torch.from_numpy(W1).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(b1, ref)
    # ties go to even: 1 + 2^-8 -> 1.0 ; 1 + 3*2^-8 -> 1 + 2^-6
    ties = np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8)], dtype=np.float32)
    assert oracle.f32_to_bf16_bits(ties).tolist() == [0x3F80, 0x3F82, 0xBF80]


def test_cosine_closed_forms():
    th = 0.7
    X = np.array([1.0, 0.0, 0.0])
    Y = np.array([math.cos(th), math.sin(th), 0.0]) * 3.0
    xy, xx, yy, c = oracle.cosine(X, Y)
    assert abs(c - math.cos(th)) < 1e-15 and abs(yy - 9.0) < 1e-14 and xx == 1.0
    assert oracle.cosine(X, X)[3] == 1.0
    assert oracle.cosine(X, np.array([0.0, 2.0, 0.0]))[3] == 0.0


def test_cosine_noise_expectation():
    """cos(G, G + sigma |G| Z / sqrt(n)) -> 1/sqrt(1 + sigma^2) for large n."""
    rng = np.random.default_rng(15)
    n = 1 << 20
    G = rng.standard_normal(n)
    for sigma in (4.0, 2.5, 1.5):
        Z = rng.standard_normal(n)
        Y = G + sigma * np.linalg.norm(G) / math.sqrt(n) * Z
        c = oracle.cosine(G, Y)[3]
        assert abs(c - 1.0 / math.sqrt(1.0 + sigma * sigma)) < 3e-3


# ---------------------------------------------------------------------------
# Post-feedforward RMSNorm (OLMo-2 / Gemma 3, Sec. 3.2 and App. E)
# ---------------------------------------------------------------------------
def _post_ffn_toy(seed, T=5, d=6, d_ff=7, V=10, small_rms_token=None, w_scale=0.3):
    rng = np.random.default_rng(seed)
    h0 = rng.standard_normal((T, d))
    A = rng.standard_normal((T, d_ff))
    W = w_scale * rng.standard_normal((d, d_ff))
    gam = 0.3 + 0.05 * rng.standard_normal(d)      # post-FFN norm weight
    w = 1.0 + 0.1 * rng.standard_normal(d)         # final norm weight
    W_U = 0.5 * rng.standard_normal((V, d))
    y = rng.integers(0, V, T).astype(np.int32)
    if small_rms_token is not None:
        A[small_rms_token] *= 0.02                 # MLP output RMS far below 0.5
    return h0, A, W, gam, w, W_U, y


def _post_ffn_loss(h0, A, Wx, gam, w, W_U, y, eps, s):
    m = A @ Wx.T                                   # MLP (down-projection) output
    rho = np.sqrt(np.mean(m * m, axis=1, keepdims=True) + eps)
    return forward_loss(h0 + gam * m / rho, w, W_U, y, eps, s)


def test_post_ffn_vjp_is_gradient_through_the_norm():
    """With a post-FFN norm and nothing above the layer, the composed signal gives
    the exact down-projection gradient: dL/dW = rmsnorm_vjp(g~, m, gamma)^T A."""
    h0, A, W, gam, w, W_U, y = _post_ffn_toy(20)
    s, eps = 1.0 / len(y), 1e-6
    m = A @ W.T
    h = h0 + gam * m / np.sqrt(np.mean(m * m, axis=1, keepdims=True) + eps)
    gt = oracle.error_signal(h, w, W_U, y, eps=eps, min_rms=0.0, s=s)["g_tilde"]
    gl = oracle.rmsnorm_vjp(gt, m, gam, eps=eps, min_rms=0.0)
    G = oracle.pseudograd(gl, A)
    fd = fd_grad(lambda Wx: _post_ffn_loss(h0, A, Wx, gam, w, W_U, y, eps, s), W.copy())
    assert rel_err(G, fd) < 1e-7


def test_post_ffn_clamp_caps_small_rms_tokens():
    """A token whose MLP output RMS is below rho_min gets (rho/rho_min) x its exact
    gradient (clamp on the 1/rho prefactor only), the others the exact one."""
    h0, A, W, gam, w, W_U, y = _post_ffn_toy(21, small_rms_token=2, w_scale=1.0)
    s, eps = 1.0, 1e-6
    m = A @ W.T
    rho = np.sqrt(np.mean(m * m, axis=1) + eps)
    assert rho[2] < 0.5 and np.all(np.delete(rho, 2) > 0.5)
    h = h0 + gam * m / rho[:, None]
    gt = oracle.error_signal(h, w, W_U, y, eps=eps, min_rms=0.5, s=s)["g_tilde"]
    exact = oracle.rmsnorm_vjp(gt, m, gam, eps=eps, min_rms=0.0)
    clamped = oracle.rmsnorm_vjp(gt, m, gam, eps=eps, min_rms=0.5)
    expect = exact.copy()
    expect[2] *= rho[2] / 0.5
    assert rel_err(clamped, expect) < 1e-14
    # the unclamped composition is the finite-difference gradient w.r.t. m
    def loss_of_m(mx):
        r = np.sqrt(np.mean(mx * mx, axis=1, keepdims=True) + eps)
        return forward_loss(h0 + gam * mx / r, w, W_U, y, eps, s)
    assert rel_err(exact, fd_grad(loss_of_m, m.copy())) < 1e-7


def test_rmsnorm_vjp_matches_error_signal_final_norm_step():
    """Applied at the final norm with the pre-VJP signal g, the standalone VJP
    reproduces the error signal's own step 5."""
    h, w, W_U, y = _toy(T=6, seed=22)
    out = oracle.error_signal(h, w, W_U, y, eps=1e-6, min_rms=0.5, s=0.3)
    again = oracle.rmsnorm_vjp(out["g"], h, w, eps=1e-6, min_rms=0.5)
    assert rel_err(again, out["g_tilde"]) < 1e-14


# ---------------------------------------------------------------------------
# Per-layer composition with the post-FFN and pre-MLP norms (Sec. 3.1 step 4, Sec. 3.2)
# ---------------------------------------------------------------------------
def _two_norm_toy(seed, T=5, d=6, V=10, small_x_token=None):
    rng = np.random.default_rng(seed)
    h0 = rng.standard_normal((T, d))
    x = rng.standard_normal((T, d))                 # input of the pre-MLP norm
    if small_x_token is not None:
        x[small_x_token] *= 0.05
    gq = 0.8 + 0.1 * rng.standard_normal(d)         # pre-MLP norm weight
    gp = 0.3 + 0.05 * rng.standard_normal(d)        # post-FFN norm weight
    w = 1.0 + 0.1 * rng.standard_normal(d)          # final norm weight
    W_U = 0.5 * rng.standard_normal((V, d))
    y = rng.integers(0, V, T).astype(np.int32)
    return h0, x, gq, gp, w, W_U, y


def _rmsn(a, eps):
    return a / np.sqrt(np.mean(a * a, axis=1, keepdims=True) + eps)


def test_layer_signal_is_gradient_through_both_norms():
    """Wire the post-FFN norm straight onto the pre-MLP norm's output (m = gq * N(x),
    h = h0 + gp * N(m)): then composing the post-FFN Jacobian at m and the pre-MLP one
    at x, in that order, is exactly dL/dx.  The other order, or a dropped norm, is not."""
    h0, x, gq, gp, w, W_U, y = _two_norm_toy(30)
    s, eps = 1.0 / len(y), 1e-6
    m = gq * _rmsn(x, eps)
    h = h0 + gp * _rmsn(m, eps)
    gt = oracle.error_signal(h, w, W_U, y, eps=eps, min_rms=0.0, s=s)["g_tilde"]
    out = oracle.layer_signal(gt, m, gp, x, gq, eps=eps, min_rms=0.0)
    fd = fd_grad(lambda xx: forward_loss(h0 + gp * _rmsn(gq * _rmsn(xx, eps), eps), w, W_U, y,
                                         eps, s), x.copy())
    assert rel_err(out, fd) < 1e-7
    swapped = oracle.rmsnorm_vjp(oracle.rmsnorm_vjp(gt, x, gq, eps=eps, min_rms=0.0), m, gp,
                                 eps=eps, min_rms=0.0)
    assert rel_err(swapped, fd) > 1e-2
    assert rel_err(oracle.layer_signal(gt, x=x, gamma_pre=gq, eps=eps, min_rms=0.0), fd) > 1e-2


def test_layer_signal_single_norm_is_that_norms_vjp():
    """With one norm the composition is that norm's App. E VJP; with none it is g."""
    h0, x, gq, gp, w, W_U, y = _two_norm_toy(31)
    rng = np.random.default_rng(32)
    g = rng.standard_normal(x.shape)
    m = rng.standard_normal(x.shape)
    assert rel_err(oracle.layer_signal(g, m, gp), oracle.rmsnorm_vjp(g, m, gp)) < 1e-15
    assert rel_err(oracle.layer_signal(g, x=x, gamma_pre=gq), oracle.rmsnorm_vjp(g, x, gq)) < 1e-15
    assert np.array_equal(oracle.layer_signal(g), g)


def test_layer_signal_clamp_acts_per_norm():
    """A token whose pre-MLP norm input has RMS below rho_min gets (rho/rho_min) x its
    unclamped signal; the post-FFN stage's clamp scales its input to the linear pre-MLP
    stage by its own factor."""
    h0, x, gq, gp, w, W_U, y = _two_norm_toy(33, small_x_token=1)
    rng = np.random.default_rng(34)
    g = rng.standard_normal(x.shape)
    m = rng.standard_normal(x.shape)
    m[3] *= 0.1                                     # post-FFN input RMS far below 0.5
    eps = 1e-6
    rx = np.sqrt(np.mean(x * x, axis=1) + eps)
    rm = np.sqrt(np.mean(m * m, axis=1) + eps)
    assert rx[1] < 0.5 and rm[3] < 0.5
    assert np.all(np.delete(rx, 1) > 0.5) and np.all(np.delete(rm, 3) > 0.5)
    exact = oracle.layer_signal(g, m, gp, x, gq, eps=eps, min_rms=0.0)
    clamped = oracle.layer_signal(g, m, gp, x, gq, eps=eps, min_rms=0.5)
    expect = exact.copy()
    expect[1] *= rx[1] / 0.5
    expect[3] *= rm[3] / 0.5
    assert rel_err(clamped, expect) < 1e-14


def test_layer_signal_eps0_is_orthogonal_to_the_pre_mlp_input():
    """With eps = 0 the last Jacobian's output is orthogonal to its norm input."""
    _, x, gq, gp, _, _, _ = _two_norm_toy(35)
    rng = np.random.default_rng(36)
    g = rng.standard_normal(x.shape)
    m = rng.standard_normal(x.shape)
    out = oracle.layer_signal(g, m, gp, x, gq, eps=0.0, min_rms=0.0)
    dots = np.abs(np.sum(out * x, axis=1)) / (np.linalg.norm(out, axis=1) * np.linalg.norm(x, axis=1))
    assert np.all(dots < 1e-13)


# ---------------------------------------------------------------------------
# Optimizers on the fp32 master and the relative clip (Sec. 3.1, App. A)
# ---------------------------------------------------------------------------
def _opt_case(seed, n=(6, 9)):
    rng = np.random.default_rng(seed)
    W = (0.02 * rng.standard_normal(n)).astype(np.float32)
    G = 1e-3 * rng.standard_normal(n)
    return W, G


def test_sgd_momentum_and_adamw_match_torch_optim():
    """Three steps against torch.optim.SGD(momentum=0.9) / AdamW(wd=0.01) in fp64."""
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(30)
    W0 = (0.02 * rng.standard_normal((5, 7))).astype(np.float32)
    grads = [1e-3 * rng.standard_normal((5, 7)) for _ in range(3)]
    for kind in (oracle.SGD_MOMENTUM, oracle.ADAMW):
        p = torch.nn.Parameter(torch.tensor(W0, dtype=torch.float64))
        opt = (torch.optim.SGD([p], lr=0.1, momentum=0.9) if kind == oracle.SGD_MOMENTUM else
               torch.optim.AdamW([p], lr=1e-3, betas=(0.9, 0.999), eps=1e-8, weight_decay=0.01))
        W, s1, s2 = W0.copy(), None, None
        for t, G in enumerate(grads, start=1):
            p.grad = torch.tensor(G)
            opt.step()
            r = oracle.optimizer_step(W, G, kind=kind, lr=0.1 if kind == oracle.SGD_MOMENTUM
                                      else 1e-3, t=t, s1=s1, s2=s2)
            # the oracle stores W and state in fp32, torch in fp64: compare to fp32 resolution
            assert np.allclose(r["W"], p.detach().numpy(), rtol=0, atol=2e-8)
            W, s1, s2 = r["W"], r["s1"], r["s2"]
            # keep torch on the same fp32-rounded trajectory
            with torch.no_grad():
                p.copy_(torch.tensor(W.astype(np.float64)))
            st = opt.state[p]
            if kind == oracle.SGD_MOMENTUM:
                assert np.allclose(s1, st["momentum_buffer"].numpy(), rtol=1e-6, atol=1e-12)
                st["momentum_buffer"].copy_(torch.tensor(s1.astype(np.float64)))
            else:
                assert np.allclose(s1, st["exp_avg"].numpy(), rtol=1e-6, atol=1e-14)
                assert np.allclose(s2, st["exp_avg_sq"].numpy(), rtol=1e-6, atol=1e-20)
                st["exp_avg"].copy_(torch.tensor(s1.astype(np.float64)))
                st["exp_avg_sq"].copy_(torch.tensor(s2.astype(np.float64)))


def test_momentum_with_zero_buffer_first_step_is_sgd():
    W, G = _opt_case(31)
    a = oracle.optimizer_step(W, G, kind=oracle.SGD_MOMENTUM, lr=0.05)
    b = oracle.optimizer_step(W, G, kind=oracle.SGD, lr=0.05)
    sg, _ = oracle.sgd_update(W, G, 0.05)
    assert np.array_equal(a["W"], b["W"]) and np.array_equal(b["W"], sg)
    assert np.array_equal(a["s1"], G.astype(np.float32))


def test_relative_clip_bounds_the_step_or_the_gradient():
    W, G = _opt_case(32)
    wn = np.linalg.norm(W.astype(np.float64))
    # update clip, active: ||W' - W|| == 0.01 ||W|| (to fp32 rounding of W')
    r = oracle.optimizer_step(W, G, kind=oracle.SGD, lr=50.0, clip=oracle.CLIP_UPDATE)
    step = r["W"].astype(np.float64) - W
    assert r["scale"] < 1 and abs(np.linalg.norm(step) - 0.01 * wn) < 1e-6 * wn
    assert rel_err(step / np.linalg.norm(step), -G / np.linalg.norm(G)) < 1e-5
    # inactive: identical to no clip
    q = oracle.optimizer_step(W, G, kind=oracle.SGD, lr=1e-3, clip=oracle.CLIP_UPDATE)
    assert q["scale"] == 1.0
    assert np.array_equal(q["W"], oracle.optimizer_step(W, G, kind=oracle.SGD, lr=1e-3)["W"])
    # gradient clip: the optimizer sees G scaled to 0.01 ||W||
    big = 10.0 * G / np.linalg.norm(G) * wn
    c = oracle.optimizer_step(W, big, kind=oracle.SGD_MOMENTUM, lr=0.1, clip=oracle.CLIP_GRADIENT)
    assert abs(np.linalg.norm(c["s1"].astype(np.float64)) - 0.01 * wn) < 1e-6 * wn
    # AdamW at t=1 with the update clip: the direction is -sign(G) - wd W / ... unchanged
    a = oracle.optimizer_step(W, G, kind=oracle.ADAMW, lr=1.0, clip=oracle.CLIP_UPDATE)
    assert abs(np.linalg.norm(a["W"].astype(np.float64) - W) - 0.01 * wn) < 1e-6 * wn


# ---------------------------------------------------------------------------
# Gate / up updates through the cached W3_init feedback (Sec. 3.1 step 5, Eq. errh)
# ---------------------------------------------------------------------------
def _silu(a):
    return a / (1.0 + np.exp(-a))


def test_gate_up_signals_are_exact_gradients_at_step_zero():
    """Nothing above the layer and W3_init = W3 (step 0, where the paper notes the
    feedback is exact): dA^T x and dB^T x are dL/dW1 and dL/dW2 of the SwiGLU MLP."""
    rng = np.random.default_rng(50)
    T, d, d_ff, V = 5, 6, 7, 9
    h0 = rng.standard_normal((T, d))
    x = rng.standard_normal((T, d))
    W1 = 0.4 * rng.standard_normal((d_ff, d))
    W2 = 0.4 * rng.standard_normal((d_ff, d))
    W3 = 0.4 * rng.standard_normal((d, d_ff))
    w = 1.0 + 0.1 * rng.standard_normal(d)
    W_U = 0.5 * rng.standard_normal((V, d))
    y = rng.integers(0, V, T).astype(np.int32)
    s, eps = 1.0 / T, 1e-6

    def loss(W1x, W2x):
        return forward_loss(h0 + (_silu(x @ W1x.T) * (x @ W2x.T)) @ W3.T, w, W_U, y, eps, s)

    a, b = x @ W1.T, x @ W2.T
    h = h0 + (_silu(a) * b) @ W3.T
    gt = oracle.error_signal(h, w, W_U, y, eps=eps, min_rms=0.0, s=s)["g_tilde"]
    dA, dB = oracle.gate_up_signals(gt, W3, a, b)
    G1 = oracle.pseudograd(dA, x)   # [d_ff, d] = dA^T x
    G2 = oracle.pseudograd(dB, x)
    fd1 = fd_grad(lambda W1x: loss(W1x, W2), W1.copy())
    fd2 = fd_grad(lambda W2x: loss(W1, W2x), W2.copy())
    assert rel_err(G1, fd1) < 1e-7
    assert rel_err(G2, fd2) < 1e-7
    # and the down-projection signal of the same layer stays g~^T h_mid
    fd3 = fd_grad(lambda W3x: forward_loss(h0 + (_silu(a) * b) @ W3x.T, w, W_U, y, eps, s),
                  W3.copy())
    assert rel_err(oracle.pseudograd(gt, _silu(a) * b), fd3) < 1e-7


def test_silu_derivative_against_autograd():
    torch = pytest.importorskip("torch")
    a = np.linspace(-8, 8, 101)
    at = torch.tensor(a, requires_grad=True)
    torch.nn.functional.silu(at).sum().backward()
    # dB / error_h = silu(a) and dA / (error_h b) = silu'(a) with error_h = b = 1
    T = 1
    g = np.ones((T, 1))
    W3 = np.ones((1, a.size))
    dA, dB = oracle.gate_up_signals(g, W3, a[None, :], np.ones((T, a.size)))
    assert np.allclose(dA[0], at.grad.numpy(), rtol=1e-12, atol=1e-14)
    assert np.allclose(dB[0], torch.nn.functional.silu(torch.tensor(a)).numpy(), rtol=1e-12,
                       atol=1e-14)


def test_norm_ratio_closed_forms_and_library_norms():
    """App. C update-magnitude ratio ||G||_F / ||W||_F: G = c W gives |c|; random arrays
    (bf16 bits and fp32) against numpy's Frobenius norms; the rate is rel / ratio."""
    rng = np.random.default_rng(11)
    W = rng.standard_normal(1000).astype(np.float32)
    out = oracle.norm_ratio([(-0.37 * W.astype(np.float64)).astype(np.float32)], [W], rel=0.01)
    assert abs(out[0, 2] - 0.37) < 1e-6 and abs(out[0, 3] - 0.01 / 0.37) < 1e-6
    Gs = [rng.standard_normal(777).astype(np.float32) * s for s in (1e-3, 2.0, 5.0)]
    Ws = [rng.standard_normal(777).astype(np.float32) for _ in range(3)]
    Gb = [oracle.f32_to_bf16_bits(g) for g in Gs]
    out = oracle.norm_ratio(Gb, Ws, rel=0.05)
    for l in range(3):
        gv = oracle.bf16_bits_to_f64(Gb[l])
        wv = Ws[l].astype(np.float64)
        assert abs(out[l, 0] - np.linalg.norm(gv) ** 2) <= 1e-12 * out[l, 0]
        assert abs(out[l, 1] - np.linalg.norm(wv) ** 2) <= 1e-12 * out[l, 1]
        r = np.linalg.norm(gv) / np.linalg.norm(wv)
        assert abs(out[l, 2] - r) <= 1e-12 * r and abs(out[l, 3] - 0.05 / r) <= 1e-12 / r
    z = oracle.norm_ratio([np.zeros(4, np.float32)], [np.ones(4, np.float32)], rel=0.01)
    assert z[0, 2] == 0.0 and math.isinf(z[0, 3])


def test_norm_ratio_reproduces_the_papers_implied_learning_rates():
    """The App. C table's implied-SGD-LR column is the 1% relative step over the ratio."""
    with open(os.path.join(GOLDEN, "update_ratio_olmo2_table.json")) as f:
        tab = json.load(f)
    for row in tab["rows"]:
        r = row["ratio_post_ffn"]
        out = oracle.norm_ratio([np.array([r, 0.0])], [np.array([0.0, 1.0])],
                                rel=tab["relative_step"])
        assert abs(out[0, 2] - r) < 1e-15
        assert round(out[0, 3], 4) == row["implied_sgd_lr"], row["layer"]
