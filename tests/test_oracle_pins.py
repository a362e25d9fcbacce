"""Pins of the fp64 oracle to facts the paper and the mathematics fix.

Each test checks the oracle against something other than itself: IEEE bit
patterns, the SVD reconstruction identity, the paper's printed kappa_b table,
the 1-bit closed form sin^2(theta) and its Gaussian limit 1 - 2/pi, brute-force
top-k, hand-evaluated SwiGLU on identity factors, and invariances.
"""
import math
import os

import numpy as np
import pytest

import oracle
import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _tiny_spec(**kw):
    base = dict(D=64, E=4, I=128, n=64, group=32, top_k=2)
    base.update(kw)
    return synth.scaled_spec(synth.WORKLOADS["tiny"], **base)


# --------------------------------------------------------------------------
def test_bit_pattern_decoding():
    bf = np.array([0x3F80, 0xC000, 0x0000, 0x4049, 0x3EAA], dtype=np.uint16)
    np.testing.assert_array_equal(oracle.bf16_bits_to_f64(bf),
                                  [1.0, -2.0, 0.0, 3.140625, 0.33203125])
    hf = np.array([0x3C00, 0x7BFF, 0xBC00, 0x0001, 0x3555], dtype=np.uint16)
    np.testing.assert_array_equal(oracle.f16_bits_to_f64(hf),
                                  [1.0, 65504.0, -1.0, 2.0 ** -24, 0.333251953125])


# --------------------------------------------------------------------------
# (a) shared basis x spectral factor reconstructs the stacked expert weights
# --------------------------------------------------------------------------
@pytest.mark.parametrize("side", ["in", "out"])
def test_shared_basis_identity(side):
    rng = np.random.default_rng(5)
    E, I, D = 3, 5, 4
    if side == "in":
        W = [rng.standard_normal((I, D)) for _ in range(E)]
    else:
        W = [rng.standard_normal((D, I)) for _ in range(E)]
    Phi, A, P = oracle.shared_basis_decompose(W, side)
    n = Phi.shape[1]
    # unit-norm normalised spectral vectors
    for e in range(E):
        np.testing.assert_allclose(np.linalg.norm(P[e], axis=0), 1.0, atol=1e-12)
    # matrix form W_e = P A Phi^T (in) / Phi A P^T (out)
    for e in range(E):
        rec = P[e] @ np.diag(A[e]) @ Phi.T if side == "in" else Phi @ np.diag(A[e]) @ P[e].T
        np.testing.assert_allclose(rec, W[e], atol=1e-12)
    # rank-one component form, summed by hand
    for e in range(E):
        acc = np.zeros_like(W[e])
        for k in range(n):
            for r in range(acc.shape[0]):
                for c in range(acc.shape[1]):
                    if side == "in":
                        acc[r, c] += A[e, k] * P[e][r, k] * Phi[c, k]
                    else:
                        acc[r, c] += A[e, k] * Phi[r, k] * P[e][c, k]
        np.testing.assert_allclose(acc, W[e], atol=1e-12)
    # energies: sum_e alpha_{e,k}^2 = sigma_k^2, sigma from a brute-force eigen solve
    Wcat = np.concatenate(W, axis=0 if side == "in" else 1)
    G = Wcat.T @ Wcat if side == "in" else Wcat @ Wcat.T
    sig2 = np.sort(np.linalg.eigvalsh(G))[::-1][:n]
    np.testing.assert_allclose(np.sum(A ** 2, axis=0), sig2, rtol=1e-10, atol=1e-10)


def _layer_from_dense(Wg, Wu, Wd):
    """Factor dense SwiGLU experts with the oracle's shared-basis decomposition and
    store them with every unit unquantised (b = 16, fp16 values; bf16 bases)."""
    E = len(Wg)
    I, D = Wg[0].shape
    layer = dict(D=D, E=E, I=I, group=I)
    bases, bits, alphas, codes = [], [], [], []
    for W, side in ((Wg, "in"), (Wu, "in"), (Wd, "out")):
        Phi, A, P = oracle.shared_basis_decompose(W, side)
        n = Phi.shape[1]
        bases.append(synth.f32_to_bf16_bits(Phi.astype(np.float32)))
        bits.append(np.full((E, n), 16, dtype=np.uint8))
        alphas.append(A.astype(np.float32))
        codes.append(np.stack([synth.f32_to_f16_bits(P[e].T.astype(np.float32)) for e in range(E)]))
    n = bases[0].shape[1]
    assert all(b.shape[1] == n for b in bases)
    layer.update(n=n, basis=np.stack(bases), bits=np.stack(bits), alpha=np.stack(alphas),
                 codes=np.stack(codes),
                 scale=np.zeros((3, E, n, 1), np.uint16), zero=np.zeros((3, E, n, 1), np.uint16))
    return layer


def test_unquantised_layer_reproduces_dense_moe():
    rng = np.random.default_rng(11)
    E, I, D, T, k = 4, 24, 16, 5, 2
    Wg = [rng.standard_normal((I, D)) * 0.5 for _ in range(E)]
    Wu = [rng.standard_normal((I, D)) * 0.5 for _ in range(E)]
    Wd = [rng.standard_normal((D, I)) * 0.5 for _ in range(E)]
    layer = _layer_from_dense(Wg, Wu, Wd)
    # weights: reconstruction within bf16 (basis) + fp16 (factor) rounding
    for e in range(E):
        g, u, d = oracle.expert_weights(layer, e)
        for got, ref in ((g, Wg[e]), (u, Wu[e]), (d, Wd[e])):
            rel = np.linalg.norm(got - ref) / np.linalg.norm(ref)
            assert rel < 1e-2, rel
    # forward against an independent dense SwiGLU MoE written from the original weights
    x_bits = synth.f32_to_bf16_bits(rng.standard_normal((T, D)).astype(np.float32))
    logits = rng.standard_normal((T, E)).astype(np.float32)
    y = oracle.moe_forward_dense(layer, x_bits, logits, k)
    x = oracle.bf16_bits_to_f64(x_bits)
    yref = np.zeros((T, D))
    for t in range(T):
        order = sorted(range(E), key=lambda e: (-float(logits[t, e]), e))[:k]
        ws = [math.exp(float(logits[t, e])) for e in order]
        for e, wgt in zip(order, ws):
            a = Wg[e] @ x[t]
            hvec = a / (1 + np.exp(-a)) * (Wu[e] @ x[t])
            yref[t] += wgt / sum(ws) * (Wd[e] @ hvec)
    err = np.max(np.abs(y - yref)) / np.max(np.abs(yref))
    assert err < 2e-2, err


# --------------------------------------------------------------------------
# (b) a 0-bit unit contributes exactly zero
# --------------------------------------------------------------------------
def test_zero_bit_unit_contributes_nothing():
    spec = _tiny_spec()
    layer = synth.make_layer(spec, seed=3)
    layer["bits"][:] = np.where(layer["bits"] == 0, 2, layer["bits"])
    x, logits = synth.make_inputs(spec, 3, seed=3)
    rng = np.random.default_rng(0)
    for h in range(3):
        for _ in range(3):
            e, j = int(rng.integers(spec.E)), int(rng.integers(spec.n))
            evicted = {k: v.copy() if isinstance(v, np.ndarray) else v for k, v in layer.items()}
            evicted["bits"][h, e, j] = 0
            # stored codes/scales of an evicted unit are irrelevant
            evicted["codes"][h, e, j] = rng.integers(0, 4, spec.I)
            evicted["scale"][h, e, j] = 0x3C00
            zero_alpha = {k: v.copy() if isinstance(v, np.ndarray) else v for k, v in layer.items()}
            zero_alpha["alpha"][h, e, j] = 0.0
            for ee in range(spec.E):
                w0 = oracle.expert_weights(evicted, ee)
                w1 = oracle.expert_weights(zero_alpha, ee)
                for a, b in zip(w0, w1):
                    np.testing.assert_array_equal(a, b)
            np.testing.assert_array_equal(
                oracle.moe_forward_factored(evicted, x, logits, spec.top_k),
                oracle.moe_forward_factored(zero_alpha, x, logits, spec.top_k))
            p = oracle.dequantize_unit(0, evicted["codes"][h, e, j], evicted["scale"][h, e, j],
                                       evicted["zero"][h, e, j], spec.group)
            assert not p.any()


# --------------------------------------------------------------------------
# symmetric quantiser: stored as codes q + 2^(b-1), zero 2^(b-1) -> exact levels
# and the paper's kappa_b table
# --------------------------------------------------------------------------
def _encode_symmetric(p, b, s):
    lv = oracle.quantize_symmetric(p, b, s)
    codes = (lv + (1 << (b - 1))).astype(np.uint16)
    scale = synth.f32_to_f16_bits(np.array([s], np.float32))
    zero = synth.f32_to_f16_bits(np.array([1 << (b - 1)], np.float32))
    return lv, codes, scale, zero


def _read_kappa():
    out = {}
    with open(os.path.join(GOLDEN, "kappa_values.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                b, v = line.split()
                out[int(b)] = float(v)
    return out


@pytest.mark.parametrize("b", [2, 3, 4, 6, 8])
def test_symmetric_levels_roundtrip_exactly(b):
    rng = np.random.default_rng(b)
    d = 256
    p = rng.standard_normal(d)
    p /= np.linalg.norm(p)
    s = float(np.float16(oracle.mse_optimal_scale(p, b, grid=200)))
    lv, codes, scale, zero = _encode_symmetric(p, b, s)
    assert codes.max() < (1 << b)
    ph = oracle.dequantize_unit(b, codes, scale, zero, d)
    np.testing.assert_array_equal(ph, s * lv)


def test_kappa_table():
    kappa = _read_kappa()
    rng = np.random.default_rng(2024)
    d, nvec = 768, 96
    P = rng.standard_normal((nvec, d))
    P /= np.linalg.norm(P, axis=1, keepdims=True)
    for b, ref in kappa.items():
        dist = []
        for p in P:
            s = oracle.mse_optimal_scale(p, b, grid=300)
            lv, codes, scale, zero = _encode_symmetric(p, b, s)
            # keep the scale exact in fp16 so the stored unit is the quantiser's output
            s16 = float(oracle.f16_bits_to_f64(scale)[0])
            lv, codes, scale, zero = _encode_symmetric(p, b, s16)
            ph = oracle.dequantize_unit(b, codes, scale, zero, d)
            dist.append(np.sum((p - ph) ** 2))
        got = float(np.mean(dist))
        assert abs(got - ref) / ref < 0.06, (b, got, ref)


# --------------------------------------------------------------------------
# 1-bit: sign quantiser stored as codes [p >= 0], zero 1/2, scale 2 s_1
# --------------------------------------------------------------------------
def _encode_sign(p):
    sg, s1 = oracle.quantize_sign(p)
    codes = (sg > 0).astype(np.uint16)
    scale = synth.f32_to_f16_bits(np.array([2 * s1], np.float32))
    zero = synth.f32_to_f16_bits(np.array([0.5], np.float32))
    return codes, scale, zero, s1


def test_one_bit_closed_form():
    rng = np.random.default_rng(7)
    d = 768
    for trial in range(20):
        p = rng.standard_normal(d)
        p[rng.integers(d)] = 0.0                 # sign(0) = +1
        p /= np.linalg.norm(p)
        codes, scale, zero, s1 = _encode_sign(p)
        ph = oracle.dequantize_unit(1, codes, scale, zero, d)
        s_st = float(oracle.f16_bits_to_f64(scale)[0]) / 2
        np.testing.assert_array_equal(ph, np.where(p >= 0, s_st, -s_st))
        # Lemma (one-bit sign distortion): ||p - Q_1(p)||^2 = sin^2(theta) = 1 - (||p||_1 / sqrt(d))^2
        sin2 = 1.0 - (np.sum(np.abs(p)) / math.sqrt(d)) ** 2
        got = np.sum((p - ph) ** 2)
        assert abs(got - sin2) < 1e-6, (got, sin2)


def test_one_bit_gaussian_limit():
    rng = np.random.default_rng(8)
    d = 4096
    vals = []
    for _ in range(50):
        p = rng.standard_normal(d)
        p /= np.linalg.norm(p)
        codes, scale, zero, _ = _encode_sign(p)
        vals.append(np.sum((p - oracle.dequantize_unit(1, codes, scale, zero, d)) ** 2))
    assert abs(np.mean(vals) - (1 - 2 / math.pi)) < 2e-3


# --------------------------------------------------------------------------
# (c) uniform bit-width: the factor is a plain group-quantised matrix
# --------------------------------------------------------------------------
@pytest.mark.parametrize("b", [1, 2, 4, 8])
def test_uniform_bits_is_group_quantised_gemv(b):
    spec = _tiny_spec()
    layer = synth.make_layer(spec, seed=9, bits_dist={b: 1.0})
    x, logits = synth.make_inputs(spec, 2, seed=9)
    xf = oracle.bf16_bits_to_f64(x)
    for h in (0, 1):
        for e in range(spec.E):
            # dense group-dequantised matrix by broadcasting whole arrays at once
            q = layer["codes"][h, e].astype(np.float64)                  # n x I
            S = np.repeat(oracle.f16_bits_to_f64(layer["scale"][h, e]), spec.group, axis=1)
            Z = np.repeat(oracle.f16_bits_to_f64(layer["zero"][h, e]), spec.group, axis=1)
            Wq = (S * (q - Z)).T                                         # I x n
            P = oracle.dequantize_factor(layer, h, e)
            np.testing.assert_array_equal(P, Wq)
            z = xf @ oracle.basis(layer, h)
            g1 = (Wq * layer["alpha"][h, e][None, :].astype(np.float64)) @ z.T
            g2 = oracle.expert_weights(layer, e)[h] @ xf.T
            np.testing.assert_allclose(g1, g2, rtol=1e-9, atol=1e-12)


# --------------------------------------------------------------------------
# (d) a consistent permutation of units leaves the output unchanged
# --------------------------------------------------------------------------
def test_unit_permutation_invariance():
    spec = _tiny_spec()
    layer = synth.make_layer(spec, seed=4)
    x, logits = synth.make_inputs(spec, 4, seed=4)
    y0 = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    perm = np.random.default_rng(1).permutation(spec.n)
    y1 = oracle.moe_forward_factored(synth.permute_units(layer, perm), x, logits, spec.top_k)
    np.testing.assert_allclose(y1, y0, rtol=1e-10, atol=1e-12 * np.abs(y0).max())
    # a permutation of the basis alone (not the units) does change it
    bad = dict(layer)
    bad["basis"] = layer["basis"][:, :, perm]
    y2 = oracle.moe_forward_factored(bad, x, logits, spec.top_k)
    assert np.max(np.abs(y2 - y0)) > 1e-3 * np.abs(y0).max()


# --------------------------------------------------------------------------
# routing: brute-force top-k with ties, softmax over the selected logits
# --------------------------------------------------------------------------
def test_routing_bruteforce():
    rng = np.random.default_rng(12)
    T, E, k = 40, 9, 3
    logits = rng.integers(-3, 4, size=(T, E)).astype(np.float32)   # many ties
    idx, w = oracle.route(logits, k)
    for t in range(T):
        ref = sorted(range(E), key=lambda e: (-float(logits[t, e]), e))[:k]
        assert list(idx[t]) == ref
        ex = [math.exp(float(logits[t, e])) for e in ref]
        np.testing.assert_allclose(w[t], np.array(ex) / sum(ex), rtol=1e-14)
        # equals softmax over all experts, then top-k, then renormalise
        full = np.exp(logits[t].astype(np.float64))
        full /= full.sum()
        np.testing.assert_allclose(w[t], full[ref] / full[ref].sum(), rtol=1e-12)


# --------------------------------------------------------------------------
# SwiGLU wiring: identity factors and bases give y = SiLU(a_g x) * (a_u x)
# --------------------------------------------------------------------------
def test_swiglu_on_identity_factors():
    D = 8
    eye_bf16 = synth.f32_to_bf16_bits(np.eye(D, dtype=np.float32))
    eye_f16 = synth.f32_to_f16_bits(np.eye(D, dtype=np.float32))
    layer = dict(D=D, E=1, I=D, n=D, group=D,
                 basis=np.stack([eye_bf16] * 3),
                 bits=np.full((3, 1, D), 16, np.uint8),
                 alpha=np.stack([np.full((1, D), a, np.float32) for a in (2.0, 3.0, 0.5)]),
                 codes=np.stack([eye_f16[None]] * 3),
                 scale=np.zeros((3, 1, D, 1), np.uint16), zero=np.zeros((3, 1, D, 1), np.uint16))
    xs = np.array([[-2.0, -1.0, -0.5, 0.0, 0.25, 0.5, 1.0, 2.0]], np.float32)
    x_bits = synth.f32_to_bf16_bits(xs)
    logits = np.zeros((1, 1), np.float32)
    expect = [0.5 * (2 * v / (1 + math.exp(-2 * v))) * (3 * v) for v in map(float, xs[0])]
    for fwd in (oracle.moe_forward_dense, oracle.moe_forward_factored):
        np.testing.assert_allclose(fwd(layer, x_bits, logits, 1)[0], expect, rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(oracle.silu(np.array([0.0, 1.0, -1.0])),
                               [0.0, 0.7310585786300049, -0.2689414213699951], rtol=1e-15)


# --------------------------------------------------------------------------
# the factored association equals the definition
# --------------------------------------------------------------------------
@pytest.mark.parametrize("alpha_scale", [1.0, 30.0])
def test_factored_equals_dense_tiny(alpha_scale):
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=0, alpha_scale=alpha_scale)
    x, logits = synth.make_inputs(spec, 4, seed=0)
    yd = oracle.moe_forward_dense(layer, x, logits, spec.top_k)
    yf = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    np.testing.assert_allclose(yf, yd, rtol=1e-9, atol=1e-11 * np.abs(yd).max())


def test_factor_matrix_matches_per_unit_definition():
    spec = _tiny_spec(n=40, I=96, group=32)
    layer = synth.make_layer(spec, seed=21, bits_dist={0: .1, 1: .15, 2: .2, 3: .15, 4: .1, 6: .1, 8: .1, 16: .1})
    for h in range(3):
        for e in range(spec.E):
            P = oracle.dequantize_factor(layer, h, e)
            for k in range(spec.n):
                col = oracle.dequantize_unit(int(layer["bits"][h, e, k]), layer["codes"][h, e, k],
                                             layer["scale"][h, e, k], layer["zero"][h, e, k], spec.group)
                np.testing.assert_array_equal(P[:, k], col)


def test_rms_norm_closed_forms():
    # constant rows: r = c / sqrt(c^2 + eps) exactly
    for c in (3.0, -0.5, 1e-3):
        h = np.full((1, 64), c)
        np.testing.assert_allclose(oracle.rms_norm(h, 1e-6), c / math.sqrt(c * c + 1e-6), rtol=1e-14)
    # any row: mean(r^2) = m / (m + eps) with m = mean(h^2); scale invariance for eps = 0
    h = np.random.default_rng(3).standard_normal((5, 100))
    m = np.mean(h * h, axis=1)
    r = oracle.rms_norm(h, 1e-2)
    np.testing.assert_allclose(np.mean(r * r, axis=1), m / (m + 1e-2), rtol=1e-12)
    np.testing.assert_allclose(oracle.rms_norm(7.0 * h, 0.0), oracle.rms_norm(h, 0.0), rtol=1e-12)


# --------------------------------------------------------------------------
# router logits of a stacked block: W_r x with W_r E x D, hand-evaluated
# --------------------------------------------------------------------------
def _bf16(vals):
    """bf16 bit patterns of values that bf16 holds exactly (the top half of their fp32 bits)."""
    return (np.asarray(vals, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def test_router_logits_hand_values():
    # one-hot router rows pick coordinates of x: logit e = x[c_e]
    x = _bf16([[1.0, -2.0, 0.5, 3.0, 0.25], [4.0, 0.0, -0.75, 1.5, 8.0]])
    pick = [3, 0, 4]
    W = np.zeros((3, 5), dtype=np.float32)
    W[np.arange(3), pick] = 1.0
    got = oracle.router_logits(_bf16(W), x)
    np.testing.assert_array_equal(got, [[3.0, 1.0, 0.25], [1.5, 4.0, 8.0]])
    # non-square (E = 2 < D = 4), sums written out by hand
    W2 = _bf16([[1.0, 2.0, 0.0, 0.0], [0.0, 0.0, -1.0, 0.5]])
    x2 = _bf16([[1.0, 1.0, 1.0, 1.0], [2.0, 1.0, 4.0, 10.0]])
    np.testing.assert_array_equal(oracle.router_logits(W2, x2), [[3.0, -0.5], [4.0, 1.0]])
    # square and not symmetric: a transposed operand gives [1, 3] instead of [3, 1]
    W3 = _bf16([[1.0, 2.0], [0.0, 1.0]])
    np.testing.assert_array_equal(oracle.router_logits(W3, _bf16([[1.0, 1.0]])), [[3.0, 1.0]])
    # the router weights are read as bf16 (0x3F81 = 1 + 2^-7), not rounded or truncated further
    W4 = np.array([[0x3F81, 0x4040]], dtype=np.uint16)            # 1.0078125, 3.0
    np.testing.assert_array_equal(oracle.router_logits(W4, _bf16([[2.0, -1.0]])), [[2.015625 - 3.0]])
