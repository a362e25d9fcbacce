"""Pins of the quantiser oracle (oracle/quantizer.py) to facts fixed by the paper
and by the mathematics, each checked against something other than the oracle:
the forward oracle's own decoder of the stored format, an fp64 evaluation of the
quantisation error with true division, the exact MSE-optimal scale found by
enumerating every breakpoint of the error on tiny groups, the paper's printed
kappa_b table, the one-bit closed form sin^2(theta) and its Gaussian limit
1 - 2/pi, fp16 rounding, and power-of-two and permutation invariances.
"""
import math
import os

import numpy as np
import pytest

import oracle
import synth
from oracle import quantizer as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
ALL_BITS = {0: .05, 1: .15, 2: .25, 3: .2, 4: .15, 6: .08, 8: .07, 16: .05}


def _decode(codes, scale, zero, bits, group):
    """p_hat of every unit through the forward oracle's decoder of the stored format."""
    return np.stack([oracle.dequantize_unit(int(b), c, s, z, group)
                     for b, c, s, z in zip(bits, codes, scale, zero)])


def _f16v(bits_u16):
    return bits_u16.view(np.float16).astype(np.float64)


def _err64(p, s, b):
    """||p - Q_b(p; s)||^2 in fp64 with true division (Eq. app_scalar_quantization_uk)."""
    qmin, qmax = -(1 << (b - 1)), (1 << (b - 1)) - 1
    q = np.clip(np.rint(p / s), qmin, qmax)
    return float(np.sum((p - s * q) ** 2))


def _exact_min_error(p, b):
    """min over s > 0 of ||p - Q_b(p; s)||^2: between consecutive breakpoints (where some
    p_i / s crosses a half-integer) the levels are fixed and the error is a quadratic in s,
    minimised at <p, q> / <q, q> clipped to the interval."""
    qmin, qmax = -(1 << (b - 1)), (1 << (b - 1)) - 1
    bps = sorted({abs(v) / (k + 0.5) for v in p if v != 0 for k in range(0, (1 << (b - 1)) + 1)})
    edges = [bps[0] * 1e-6] + bps + [bps[-1] * 10.0]
    best = float(np.dot(p, p))
    for lo, hi in zip(edges[:-1], edges[1:]):
        q = np.clip(np.rint(p / (0.5 * (lo + hi))), qmin, qmax)
        qq = float(np.dot(q, q))
        if qq == 0:
            continue
        s = min(max(float(np.dot(p, q)) / qq, lo), hi)
        best = min(best, float(np.sum((p - s * q) ** 2)))
    return best


# --------------------------------------------------------------------------
@pytest.mark.parametrize("b", [2, 3, 4, 6, 8])
def test_stored_units_decode_to_symmetric_levels_within_half_a_step(b):
    P, _ = synth.make_float_units(24, 256, seed=b)
    bits = np.full(24, b, np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=64)
    ph = _decode(codes, scale, zero, bits, 64)
    s = np.repeat(_f16v(scale), 64, axis=1)
    assert np.all(_f16v(zero) == 2.0 ** (b - 1))
    assert codes.max() < (1 << b)
    lv = ph / s
    np.testing.assert_array_equal(lv, np.rint(lv))                   # integer levels
    assert lv.min() >= -(1 << (b - 1)) and lv.max() <= (1 << (b - 1)) - 1
    p = P.astype(np.float64)
    inside = np.abs(p) <= s * ((1 << (b - 1)) - 0.5)                 # not clipped
    tol = 1e-6 * s
    assert np.all(np.abs(p - ph)[inside] <= s[inside] / 2 + tol[inside])
    # the clipped ones sit on an end level and only beyond it
    assert np.all((np.abs(lv) >= (1 << (b - 1)) - 1)[~inside])


@pytest.mark.parametrize("b", [2, 3, 4])
def test_search_picks_the_least_error_candidate(b):
    P, _ = synth.make_float_units(16, 512, seed=10 + b)
    bits = np.full(16, b, np.uint8)
    g = 128
    _, scale, _ = Q.quantize_units(P, bits, group=g, grid=256)
    s_got = _f16v(scale)
    for u in range(16):
        for gi in range(512 // g):
            p = P[u, gi * g:(gi + 1) * g].astype(np.float64)
            top = np.abs(p).max() * 2.0 ** (2 - b)
            cands = np.float16(np.float32(np.float32(top) * np.arange(1, 257, dtype=np.float32))
                               / np.float32(256)).astype(np.float64)
            errs = [_err64(p, s, b) for s in cands if s > 0]
            got = _err64(p, s_got[u, gi], b)
            assert got <= min(errs) * (1 + 1e-5) + 1e-12, (u, gi, got, min(errs))


@pytest.mark.parametrize("b", [2, 3, 4])
def test_search_is_near_the_exact_mse_optimum(b):
    rng = np.random.default_rng(50 + b)
    g = 32
    P = rng.standard_normal((40, g)).astype(np.float32)
    P /= np.linalg.norm(P, axis=1, keepdims=True)
    bits = np.full(40, b, np.uint8)
    _, scale, _ = Q.quantize_units(P, bits, group=g, grid=256)
    for u in range(40):
        p = P[u].astype(np.float64)
        exact = _exact_min_error(p, b)
        got = _err64(p, float(_f16v(scale)[u, 0]), b)
        assert got >= exact - 1e-12                                   # nothing beats the optimum
        assert got <= exact * 1.02 + 1e-9, (u, got, exact)            # the grid gets within 2 %


def _read_kappa():
    out = {}
    with open(os.path.join(GOLDEN, "kappa_values.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                out[int(k)] = float(v)
    return out


def test_kappa_table_with_one_scale_per_vector():
    """Table kappa_values: mean ||p - Q_b(p)||^2 of unit-norm vectors with the MSE-optimal
    per-vector scale (the quantiser of the appendix analysis: one group = the whole vector)."""
    kappa = _read_kappa()
    d, nvec = 768, 96
    P, _ = synth.make_float_units(nvec, d, seed=2024)
    for b, ref in kappa.items():
        bits = np.full(nvec, b, np.uint8)
        codes, scale, zero = Q.quantize_units(P, bits, group=d, grid=512)
        ph = _decode(codes, scale, zero, bits, d)
        got = float(np.mean(np.sum((P.astype(np.float64) - ph) ** 2, axis=1)))
        assert abs(got - ref) / ref < 0.06, (b, got, ref)
    # finer groups (the stored format, group 128) only lower the distortion
    bits = np.full(nvec, 2, np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=128)
    ph = _decode(codes, scale, zero, bits, 128)
    assert float(np.mean(np.sum((P.astype(np.float64) - ph) ** 2, axis=1))) < kappa[2]


def test_one_bit_sign_quantiser_closed_form_and_gaussian_limit():
    d = 768
    P, _ = synth.make_float_units(200, d, seed=7)
    P[0, 5] = 0.0
    P[1, 9] = -0.0                                                    # sign(0) = +1 for either zero
    bits = np.ones(200, np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=d)
    p64 = P.astype(np.float64)
    np.testing.assert_array_equal(codes, (p64 >= 0).astype(np.uint16))
    assert codes[0, 5] == 1 and codes[1, 9] == 1
    assert np.all(_f16v(zero) == 0.5)
    s1 = np.mean(np.abs(p64), axis=1)
    np.testing.assert_allclose(_f16v(scale)[:, 0] / 2, s1, rtol=2.0 ** -11)
    ph = _decode(codes, scale, zero, bits, d)
    dist = np.sum((p64 - ph) ** 2, axis=1)
    # Lemma (one-bit sign distortion) at the stored scale s: ||p - s sign p||^2 =
    # ||p||^2 - 2 s ||p||_1 + d s^2, which is ||p||^2 sin^2(theta) = ||p||^2 - ||p||_1^2 / d at
    # s = s_1 (rows 0 and 1 lost an element after normalisation, so ||p|| is not 1 there)
    s = _f16v(scale)[:, 0] / 2
    l1 = np.sum(np.abs(p64), axis=1)
    l2 = np.sum(p64 * p64, axis=1)
    np.testing.assert_allclose(dist, l2 - 2 * s * l1 + d * s * s, rtol=1e-9, atol=1e-12)
    np.testing.assert_allclose(dist, l2 - l1 ** 2 / d, rtol=0, atol=2e-6)
    assert abs(float(np.mean(dist)) - (1 - 2 / math.pi)) < 0.01


@pytest.mark.parametrize("b", [6, 8])
def test_high_bits_scale_is_max_abs_over_qmax(b):
    P, _ = synth.make_float_units(20, 256, seed=60 + b)
    bits = np.full(20, b, np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=128)
    qmax = (1 << (b - 1)) - 1
    for u in range(20):
        for gi in range(2):
            p = P[u, gi * 128:(gi + 1) * 128].astype(np.float64)
            s = float(_f16v(scale)[u, gi])
            assert s == float(np.float16(np.float32(np.abs(p).max()) / np.float32(qmax)))
            i = int(np.argmax(np.abs(p)))
            lv = int(codes[u, gi * 128 + i]) - (1 << (b - 1))
            assert abs(lv) == qmax                                    # rho lands on the end level
            ph = s * (codes[u, gi * 128:(gi + 1) * 128].astype(np.float64) - (1 << (b - 1)))
            assert np.max(np.abs(p - ph)) <= s / 2 * (1 + 1e-6)       # never clipped


def test_sixteen_and_zero_bits():
    P, _ = synth.make_float_units(6, 128, seed=3)
    P[0, :4] = [1e5, -1e-9, 65519.0, 3.0]                             # overflow, subnormal, ties
    bits = np.array([16, 0, 16, 0, 16, 0], np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=64)
    for u in (0, 2, 4):
        np.testing.assert_array_equal(codes[u], P[u].astype(np.float16).view(np.uint16))
    assert codes[0, 0] == 0x7C00 and codes[0, 2] == 0x7BFF            # +inf, 65504 (fp16 rounding)
    assert not codes[1::2].any() and not scale.any() and not zero.any()


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8])
def test_power_of_two_scaling_is_exact(b):
    P, _ = synth.make_float_units(12, 256, seed=70 + b)
    bits = np.full(12, b, np.uint8)
    c0, s0, z0 = Q.quantize_units(P, bits, group=64)
    for k in (-3, 2):
        c1, s1, z1 = Q.quantize_units(P * np.float32(2.0 ** k), bits, group=64)
        np.testing.assert_array_equal(c1, c0)
        np.testing.assert_array_equal(z1, z0)
        np.testing.assert_array_equal(_f16v(s1), _f16v(s0) * 2.0 ** k)


def test_unit_permutation_permutes_outputs():
    P, bits = synth.make_float_units(30, 256, seed=5, bits_dist=ALL_BITS)
    perm = np.random.default_rng(1).permutation(30)
    a = Q.quantize_units(P, bits, group=64)
    b = Q.quantize_units(P[perm], bits[perm], group=64)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x[perm], y)


def test_zero_groups_store_the_zero_level():
    P, _ = synth.make_float_units(8, 128, seed=9)
    P[:, :64] = 0.0
    for b in (1, 2, 3, 4, 6, 8):
        bits = np.full(8, b, np.uint8)
        codes, scale, zero = Q.quantize_units(P, bits, group=64)
        assert not _f16v(scale)[:, 0].any()
        want = 1 if b == 1 else 1 << (b - 1)
        assert np.all(codes[:, :64] == want)
        assert not _decode(codes, scale, zero, bits, 64)[:, :64].any()


def test_rejects_bad_arguments():
    P, _ = synth.make_float_units(4, 128, seed=1)
    with pytest.raises(ValueError):
        Q.quantize_units(P, np.array([2, 5, 2, 2], np.uint8), group=64)
    with pytest.raises(ValueError):
        Q.quantize_units(P, np.full(4, 2, np.uint8), group=96)


def test_quantised_layer_forward_tracks_the_float_layer():
    """A tiny layer quantised at 8 bits from float units: the forward oracle on the stored
    layer stays close to the same layer with the float units (distortion ~ 2^-16)."""
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=64, E=4, I=128, n=64, group=32, top_k=2)
    layer = synth.make_layer(spec, seed=2)
    U = 3 * spec.E * spec.n
    P, _ = synth.make_float_units(U, spec.I, seed=2)
    bits = np.full(U, 8, np.uint8)
    codes, scale, zero = Q.quantize_units(P, bits, group=spec.group)
    q = dict(layer, bits=bits.reshape(3, spec.E, spec.n),
             codes=codes.reshape(3, spec.E, spec.n, spec.I),
             scale=scale.reshape(3, spec.E, spec.n, -1), zero=zero.reshape(3, spec.E, spec.n, -1))
    f = dict(q, bits=np.full((3, spec.E, spec.n), 16, np.uint8),
             codes=P.astype(np.float16).view(np.uint16).reshape(3, spec.E, spec.n, spec.I))
    x, logits = synth.make_inputs(spec, 3, seed=2)
    yq = oracle.moe_forward_dense(q, x, logits, spec.top_k)
    yf = oracle.moe_forward_dense(f, x, logits, spec.top_k)
    assert np.max(np.abs(yq - yf)) / np.max(np.abs(yf)) < 2e-2
