"""Pins of the calibration oracle (oracle/calibration.py): the activation metric
H = X Diag(g) X^T and the importance beta of Eq. app_unified_beta_def, against closed forms
(identity and rank-one activations, Parseval's trace identity for an orthonormal basis),
homogeneity and token-order invariance, and the paper's loss itself: evicting one unit
changes the projection's g-weighted output energy by exactly alpha^2 |p|^2 beta (gate, up)
or alpha^2 |phi|^2 beta (down), computed through the forward oracle's dense weights."""
import numpy as np
import pytest

import oracle
import synth
from oracle import calibration as C


def _orthonormal(D, n, seed):
    q, _ = np.linalg.qr(np.random.default_rng(seed).standard_normal((D, n)))
    return q


def test_identity_and_rank_one_activations():
    Phi = _orthonormal(16, 16, 1)
    np.testing.assert_allclose(C.importance(Phi, C.activation_metric(np.eye(16), np.ones(16))), 1.0, rtol=1e-12)
    x = np.random.default_rng(2).standard_normal(16)
    b = C.importance(Phi, C.activation_metric(x[:, None], [1.0]))
    np.testing.assert_allclose(b, (Phi.T @ x) ** 2, rtol=1e-12)
    V = np.random.default_rng(3).standard_normal((16, 5))       # any vectors: beta = v^T H v
    H = C.activation_metric(np.eye(16), np.ones(16))
    np.testing.assert_allclose(C.importance(V, H), np.sum(V * V, axis=0), rtol=1e-12)


def test_parseval_trace_identity_and_sign():
    rng = np.random.default_rng(4)
    D, T = 24, 50
    Phi = _orthonormal(D, D, 5)
    X = rng.standard_normal((D, T))
    g = rng.uniform(0, 1, T)
    b = C.importance(Phi, C.activation_metric(X, g))
    assert np.all(b >= 0)
    np.testing.assert_allclose(b.sum(), np.sum(g * np.sum(X * X, axis=0)), rtol=1e-10)


def test_homogeneity_and_token_order():
    rng = np.random.default_rng(6)
    Phi = _orthonormal(12, 8, 7)
    X, g = rng.standard_normal((12, 30)), rng.uniform(0, 1, 30)
    b = C.importance(Phi, C.activation_metric(X, g))
    np.testing.assert_allclose(C.importance(Phi, C.activation_metric(3 * X, g)), 9 * b, rtol=1e-12)
    np.testing.assert_allclose(C.importance(Phi, C.activation_metric(X, 0.25 * g)), 0.25 * b, rtol=1e-12)
    perm = rng.permutation(30)
    np.testing.assert_allclose(C.importance(Phi, C.activation_metric(X[:, perm], g[perm])), b, rtol=1e-12)


def test_affinities_are_the_forward_gate_weights():
    logits = np.random.default_rng(8).standard_normal((9, 6)).astype(np.float32)
    g = C.affinities(logits, 2, 6)
    idx, w = oracle.route(logits, 2)
    assert np.all((g > 0).sum(axis=1) == 2)
    np.testing.assert_allclose(g.sum(axis=1), 1.0, rtol=1e-12)
    for t in range(9):
        np.testing.assert_allclose(g[t, idx[t]], w[t], rtol=0)


@pytest.mark.parametrize("h", [oracle.GATE, oracle.UP, oracle.DOWN])
def test_evicting_a_unit_costs_alpha_squared_beta(h):
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=32, E=3, I=64, n=32, group=32, top_k=2)
    layer = synth.make_layer(spec, seed=9, bits_dist={2: .3, 3: .3, 4: .2, 8: .2})
    x, logits = synth.make_inputs(spec, 40, seed=9)
    beta = C.layer_importance(layer, x, logits, spec.top_k)
    g = C.affinities(logits, spec.top_k, spec.E)
    X = oracle.bf16_bits_to_f64(x).T
    for e in range(spec.E):
        W = oracle.expert_weights(layer, e)
        Hin = C.intermediate(layer, x, e) if h == oracle.DOWN else X
        P = oracle.dequantize_factor(layer, h, e)
        Phi = oracle.basis(layer, h)
        for k in (0, 7, 31):
            ev = dict(layer, bits=layer["bits"].copy())
            ev["bits"][h, e, k] = 0
            dW = W[h] - oracle.expert_weights(ev, e)[h]
            loss = float(np.sum(g[:, e] * np.sum((dW @ Hin) ** 2, axis=0)))
            a = oracle.alpha(layer, h, e)[k]
            norm2 = float(P[:, k] @ P[:, k]) if h != oracle.DOWN else float(Phi[:, k] @ Phi[:, k])
            assert loss == pytest.approx(a * a * norm2 * beta[h, e, k], rel=1e-9, abs=1e-15)


def test_intermediate_activations_rebuild_the_forward():
    """The down projection's inputs h_{t,e}: sum_e g_{t,e} W_dn,e h_{t,e} is the MoE output of
    the forward oracle's dense definition (itself pinned by the SwiGLU wiring tests)."""
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=32, E=4, I=64, n=32, group=32, top_k=2)
    layer = synth.make_layer(spec, seed=10)
    x, logits = synth.make_inputs(spec, 12, seed=10)
    g = C.affinities(logits, spec.top_k, spec.E)
    y = np.zeros((12, spec.D))
    for e in range(spec.E):
        Wdn = oracle.expert_weights(layer, e)[2]
        y += g[:, e][:, None] * (Wdn @ C.intermediate(layer, x, e)).T
    ref = oracle.moe_forward_dense(layer, x, logits, spec.top_k)
    np.testing.assert_allclose(y, ref, rtol=1e-9, atol=1e-12 * np.max(np.abs(ref)))


def test_float_factor_importance_against_dense_weights():
    """beta from the decomposition's float factors (before quantisation): for gate/up it is
    sum_t g_t (phi_k^T x_t)^2, and for down, removing unit k of the float down factor changes
    the g-weighted output energy by alpha_k^2 beta_k, with the expert's SwiGLU activations
    taken from the dense float weights themselves (not through the factors)."""
    rng = np.random.default_rng(12)
    D, I, E, T, k = 6, 5, 3, 20, 2
    Wg = [rng.standard_normal((I, D)) for _ in range(E)]
    Wu = [rng.standard_normal((I, D)) for _ in range(E)]
    Wd = [rng.standard_normal((D, I)) for _ in range(E)]
    dec = [oracle.shared_basis_decompose(W, side) for W, side in ((Wg, "in"), (Wu, "in"), (Wd, "out"))]
    Phi = [d[0] for d in dec]
    al = [d[1] for d in dec]
    P = [d[2] for d in dec]
    x = synth.f32_to_bf16_bits(rng.standard_normal((T, D)).astype(np.float32))
    logits = rng.standard_normal((T, E)).astype(np.float32)
    beta = C.factor_importance(Phi, al, P, x, logits, k)
    g = C.affinities(logits, k, E)
    X = oracle.bf16_bits_to_f64(x).T
    for e in range(E):
        for h in (oracle.GATE, oracle.UP):
            want = np.sum(g[:, e][None, :] * (Phi[h].T @ X) ** 2, axis=1)
            np.testing.assert_allclose(beta[h, e], want, rtol=1e-10, atol=1e-12)
        Hact = oracle.silu(Wg[e] @ X) * (Wu[e] @ X)                       # I x T, dense definition
        for j in range(Phi[2].shape[1]):
            dW = al[2][e, j] * np.outer(Phi[2][:, j], P[2][e][:, j])
            loss = float(np.sum(g[:, e] * np.sum((dW @ Hact) ** 2, axis=0)))
            assert loss == pytest.approx(al[2][e, j] ** 2 * beta[2, e, j], rel=1e-9, abs=1e-12)
