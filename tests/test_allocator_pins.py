"""Pins of the bit-allocation oracle (oracle/allocator.py), each against something
other than the oracle: hand-evaluated budgets of Eq. app_projection_normalized_budget,
fp64 closed forms of the piecewise distortion, the measured one-bit distortion of the
quantiser oracle, an independent fp64 convex hull, the exact ILP optimum by dynamic
programming (the Lagrangian solution is optimal at the bits it uses) and the LP bound.
"""
import math
import os

import numpy as np
import pytest

import synth
from oracle import allocator as A
from oracle import quantizer as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _kappa():
    out = {}
    with open(os.path.join(GOLDEN, "kappa_values.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                out[int(k)] = float(v)
    return out


def test_projection_budget_by_hand():
    # Qwen3-30B-A3B shapes: 128 * 2048 * 2 - 16 * 2048^2 / 768 = 524288 - 87381.33...
    assert A.projection_budget(128, 2048, 768, 2.0) == 436906
    # Mixtral-8x7B shapes: 8 * 4096 * 2 - 16 * 4096^2 / 14336 = 65536 - 18724.57...
    assert A.projection_budget(8, 4096, 14336, 2.0) == 46811
    # 2.5 bits: 655360 - 87381.33... ; exact integers stay exact
    assert A.projection_budget(128, 2048, 768, 2.5) == 567978
    assert A.projection_budget(4, 16, 64, 3) == 4 * 16 * 3 - 64


def test_distortion_closed_forms():
    kappa = _kappa()
    P, _ = synth.make_float_units(40, 768, seed=1)
    E = A.distortion(P, kappa).astype(np.float64)
    p = P.astype(np.float64)
    d = p.shape[1]
    assert np.all(E[:, 0] == 1.0)
    np.testing.assert_allclose(E[:, 1], 1 - np.sum(np.abs(p), axis=1) ** 2 / d, rtol=0, atol=2e-6)
    for j, b in ((2, 2), (3, 3), (4, 4)):
        assert np.all(E[:, j] == np.float32(kappa[b]))
    eta = d * np.max(np.abs(p), axis=1) ** 2 / 3
    for j, b in ((5, 6), (6, 8), (7, 16)):
        np.testing.assert_allclose(E[:, j], eta * np.exp(-2 * math.log(2) * b), rtol=1e-6)


def test_one_bit_distortion_is_the_sign_quantisers_error():
    """E(1) = sin^2(theta) is the measured ||p - Q_1(p)||^2 of the sign quantiser (one
    scale for the whole vector; the stored scale is fp16-rounded)."""
    P, _ = synth.make_float_units(30, 512, seed=2)
    codes, scale, zero = Q.quantize_units(P, np.ones(30, np.uint8), group=512)
    s = scale.view(np.float16).astype(np.float64)[:, 0] / 2
    ph = np.where(codes > 0, 1.0, -1.0) * s[:, None]
    meas = np.sum((P.astype(np.float64) - ph) ** 2, axis=1)
    E1 = A.distortion(P, _kappa())[:, 1].astype(np.float64)
    np.testing.assert_allclose(E1, meas, rtol=2e-3)


def test_importance_weight():
    rng = np.random.default_rng(3)
    a = rng.uniform(0.1, 2, 50).astype(np.float32)
    b = rng.lognormal(0, 1, 50).astype(np.float32)
    a64, b64 = a.astype(np.float64), b.astype(np.float64)
    np.testing.assert_allclose(A.importance_weight(a, b, 0.0), a64 ** 2, rtol=1e-6)
    np.testing.assert_allclose(A.importance_weight(a, b, 1.0), a64 ** 2 * b64, rtol=1e-6)
    np.testing.assert_allclose(A.importance_weight(a, b, 0.5), a64 ** 2 * np.sqrt(b64), rtol=1e-6)
    with pytest.raises(ValueError):
        A.importance_weight(a, b, 0.7)


def _random_costs(rng, U):
    """Decreasing-ish random costs per unit (C(0) largest), like w E(b)."""
    w = rng.lognormal(0, 1, U)
    E = np.sort(rng.uniform(0, 1, (U, 8)), axis=1)[:, ::-1].copy()
    E[:, 0] = 1.0
    E[:, 1:] *= rng.uniform(0.2, 1.0, (U, 1))
    return (w[:, None] * E).astype(np.float32)


def _hull64(c):
    """Lower convex hull of (b, c_b) from b = 0, by Andrew's monotone chain in fp64, then
    cut where the cost stops decreasing."""
    pts = [(float(b), float(v)) for b, v in zip(A.BITS, c)]
    hull = []
    for p in pts:
        while len(hull) >= 2:
            (x1, y1), (x2, y2) = hull[-2], hull[-1]
            if (x2 - x1) * (p[1] - y1) - (y2 - y1) * (p[0] - x1) <= 0:
                hull.pop()
            else:
                break
        hull.append(p)
    out = [hull[0]]
    for p in hull[1:]:
        if p[1] < out[-1][1]:
            out.append(p)
        else:
            break
    return [int(x) for x, _ in out[1:]]


def test_hull_matches_an_independent_convex_hull():
    rng = np.random.default_rng(4)
    C = _random_costs(rng, 300)
    keys, reach = A.hull_increments(C)
    for u in range(300):
        got = [A.BITS[j] for j in reach[u] if j >= 0]
        assert got == _hull64(C[u]), (u, got, _hull64(C[u]))
        k = keys[u][keys[u] > 0]
        assert np.all(np.diff(k.astype(np.float64)) <= 0)        # efficiencies never increase
        assert np.all((k & np.uint64(0xFFFFFFFF)) == 0xFFFFFFFF - u)


@pytest.mark.parametrize("seed", range(6))
def test_lagrangian_solution_is_optimal_at_its_own_bits(seed):
    """Every prefix-closed set of hull increments taken in descending efficiency is an exact
    ILP optimum for the bits it uses; the fill keeps feasibility and never costs more, and
    nothing beats the ILP optimum or the LP bound."""
    rng = np.random.default_rng(100 + seed)
    U = int(rng.integers(3, 8))
    C = _random_costs(rng, U)
    top = int(sum(max(A.BITS[j] for j in r if j >= 0) if (r >= 0).any() else 0
                  for r in A.hull_increments(C)[1]))
    for B in range(0, top + 3):
        thr = A.allocate(C, B, fill=False)
        used = int(thr.astype(np.int64).sum())
        opt_used, _ = A.ilp_optimum(C, used)
        assert A.total_cost(C, thr) == pytest.approx(opt_used, rel=1e-6, abs=1e-9)
        # step 3 is maximal: the next group of equal keys does not fit the bits left
        keys, reach = A.hull_increments(C)
        bits = np.array(A.BITS)
        taken = np.array([int(np.sum(reach[u] >= 0)) if thr[u] == bits[reach[u][reach[u] >= 0]].max(initial=0)
                          else int(np.argmax(bits[np.maximum(reach[u], 0)] == thr[u])) + 1 for u in range(U)])
        taken = np.where(thr == 0, 0, taken)
        nxt = [(keys[u, taken[u]], u) for u in range(U) if taken[u] < 7 and keys[u, taken[u]] > 0]
        if nxt:
            kmax = max(k for k, _ in nxt)
            prev_b = np.concatenate([[0], bits[np.maximum(reach[0], 0)]])
            grp = 0
            for u in range(U):
                for i in range(taken[u], 7):
                    if keys[u, i] == kmax:
                        lo = 0 if i == 0 else bits[reach[u, i - 1]]
                        grp += bits[reach[u, i]] - lo
            assert grp > B - used, (B, used, grp)
        full = A.allocate(C, B)
        assert int(full.astype(np.int64).sum()) <= B
        opt, _ = A.ilp_optimum(C, B)
        got = A.total_cost(C, full)
        assert got <= A.total_cost(C, thr) + 1e-12
        assert got >= opt - 1e-6 * abs(opt) - 1e-9
        assert opt >= A.lp_bound(C, B) - 1e-6 * abs(opt) - 1e-9


def test_budget_extremes():
    rng = np.random.default_rng(5)
    C = _random_costs(rng, 50)
    assert not A.allocate(C, 0).any()
    big = A.allocate(C, 10 ** 6)
    # every unit at its cheapest option (the end of its hull; ties to the larger b)
    cheapest = np.array(A.BITS)[7 - np.argmin(C[:, ::-1], axis=1)]
    np.testing.assert_array_equal(big, cheapest)


def test_synthetic_layer_allocation_meets_the_budget_and_orders_by_energy():
    """Qwen3-shaped units with alpha_j = j^-1/2 and one beta per unit: the budget is met
    within the largest increment, and higher-energy units never get fewer bits on average."""
    U, I, n = 4096, 768, 2048
    P, _ = synth.make_float_units(U, I, seed=6)
    alpha = (np.arange(U) % n + 1.0) ** -0.5
    beta = np.ones(U, np.float32)
    C = A.costs(P, alpha.astype(np.float32), beta, 1.0, _kappa())
    B = int(1.67 * U)
    b = A.allocate(C, B).astype(np.int64)
    assert B - 16 < b.sum() <= B
    hi = b[(np.arange(U) % n) < n // 4].mean()
    lo = b[(np.arange(U) % n) >= 3 * n // 4].mean()
    assert hi > lo


def test_collinear_options_stay_separate_increments():
    """Options on one line (C(b) = 8 - b up to 8 bits) are equally efficient: with ties to the
    smaller b they remain unit steps, so a budget of 4 reaches b = 4 (cost 4), which the
    exact optimum confirms; a single 8-bit step could not be used at all."""
    C = np.array([[8, 7, 6, 5, 4, 2, 0, -4]], np.float32)
    keys, reach = A.hull_increments(C)
    assert [A.BITS[j] for j in reach[0] if j >= 0] == [1, 2, 3, 4, 6, 8, 16]
    for B in range(0, 20):
        b = A.allocate(C, B)
        opt, _ = A.ilp_optimum(C, B)
        assert A.total_cost(C, b) == pytest.approx(opt), (B, b, opt)

