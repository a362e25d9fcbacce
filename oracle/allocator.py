"""CPU oracle of the per-projection bit allocation (which bit-width each unit gets).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: imported by tests/ and
by the CPU legs of bench.py, never by the CUDA library or its binding, and it
shares no code with them.

What the paper defines (appendix "Component-wise Loss and ILP Formulation" and
"Piecewise Reconstruction Error for Bit Allocation"): for one projection type,
choose b_u in B = {0, 1, 2, 3, 4, 6, 8, 16} for every unit u to

    minimise  sum_u C_u(b_u)   subject to  sum_u b_u <= B_h        (Eq. ilp_piecewise_eps)

with C_u(b) = alpha_u^2 beta_u^gamma E_u(b) (Eq. app_component_loss_final) and
the piecewise distortion E_u(b) of Eq. piecewise_expected_eps:
    b in {6, 8, 16}: eta_u exp(-lambda b), eta_u = d rho_u^2 / 3, rho_u = ||p_u||_inf,
                     lambda = 2 ln 2, so exp(-lambda b) = 2^(-2b);
    b in {2, 3, 4}:  kappa_b (Table kappa_values);
    b = 1:           sin^2(theta_u) = 1 - ||p_u||_1^2 / d (Lemma one-bit sign distortion);
    b = 0:           1.
B_h = floor(E n b_eq - 16 n^2 / m) (Eq. app_projection_normalized_budget).

The paper solves the ILP with a commercial solver.  This build solves it with
the Lagrangian relaxation of the multiple-choice knapsack plus a greedy fill,
the same steps on both sides (``allocate``), and checks the result against the
exact optimum (``ilp_optimum``: dynamic programming over the budget, tiny
inputs) and the LP bound.  Steps (readings where the paper leaves the arithmetic open):

1. costs in fp32, each operation rounded once: ||p||_1 as the exact integer sum
   of floor(|p_i| 2^40) scaled by 2^-40 (order-free), sin^2 = 1 - (l1 l1) / d,
   eta = ((rho rho) d) / 3, E(b) = eta 2^(-2b), w = (alpha alpha) beta^gamma
   (beta^gamma: 1, sqrt(beta) or beta for gamma = 0, 1/2, 1), C(b) = w E(b);
2. per unit, the lower convex hull of (b, C(b)) from b = 0: from the current
   point, the next is the larger b' with the largest efficiency
   e = (C_cur - C(b')) / (b' - b_cur) > 0 (ties to the smaller b', so
   collinear options stay separate increments of equal efficiency), each
   efficiency capped at the previous one (so they never increase);
   the increment's key is (bits of e) * 2^32 + (2^32 - 1 - u);
3. take increments in descending key order while the bits stay within B_h
   (a group of equal keys is taken whole or not at all); this is the
   Lagrangian solution for the multiplier at the first increment left out;
4. greedy fill: while some unit's next increment fits the remaining bits,
   take the one with the largest key.
"""
from __future__ import annotations

from fractions import Fraction
from typing import Dict, Sequence, Tuple

import numpy as np

BITS = (0, 1, 2, 3, 4, 6, 8, 16)
F32 = np.float32
FIX_SHIFT = 40


def projection_budget(E: int, n: int, m: int, b_eq) -> int:
    """B_h = floor(E n b_eq - 16 n^2 / m) (Eq. app_projection_normalized_budget), exactly.
    Negative when the fp16 bases alone exceed the layer's budget (tiny layers): no
    allocation meets it."""
    return int(np.floor(Fraction(E * n) * Fraction(str(b_eq)) - Fraction(16 * n * n, m)))


def distortion(P: np.ndarray, kappa: Dict[int, float]) -> np.ndarray:
    """E_u(b) for every unit (rows of P, length d) and b in BITS, fp32 (U x 8)."""
    P = np.ascontiguousarray(P, dtype=F32)
    U, d = P.shape
    a = np.abs(P)
    rho = a.max(axis=1) if d else np.zeros(U, F32)
    fix = np.floor(a.astype(np.float64) * float(2 ** FIX_SHIFT)).astype(np.int64)
    l1 = fix.sum(axis=1).astype(F32) * F32(2.0 ** -FIX_SHIFT)
    sin2 = F32(1.0) - (l1 * l1) / F32(d)
    eta = ((rho * rho) * F32(d)) / F32(3.0)
    out = np.empty((U, 8), F32)
    out[:, 0] = F32(1.0)
    out[:, 1] = sin2
    out[:, 2] = F32(kappa[2])
    out[:, 3] = F32(kappa[3])
    out[:, 4] = F32(kappa[4])
    out[:, 5] = eta * F32(2.0 ** -12)
    out[:, 6] = eta * F32(2.0 ** -16)
    out[:, 7] = eta * F32(2.0 ** -32)
    return out


def importance_weight(alpha: np.ndarray, beta: np.ndarray, gamma: float) -> np.ndarray:
    """w = alpha^2 beta^gamma in fp32 (Eq. app_component_loss_final's factor), gamma in {0, 1/2, 1}."""
    a = np.asarray(alpha, F32)
    b = np.asarray(beta, F32)
    if gamma == 0.0:
        bg = np.ones_like(b)
    elif gamma == 0.5:
        bg = np.sqrt(b)
    elif gamma == 1.0:
        bg = b
    else:
        raise ValueError("the oracle's weights are exact for gamma in {0, 1/2, 1}")
    return (a * a) * bg


def costs(P, alpha, beta, gamma, kappa) -> np.ndarray:
    """C_u(b) = w_u E_u(b), fp32, U x 8."""
    return importance_weight(alpha, beta, gamma)[:, None] * distortion(P, kappa)


def hull_increments(C: np.ndarray) -> Tuple[np.ndarray, np.ndarray]:
    """Per unit, the hull increments (step 2): keys (U x 7 uint64, 0 = none) and the bit-width
    index reached by each (U x 7, -1 = none)."""
    C = np.asarray(C, F32)
    U = C.shape[0]
    bits = np.array(BITS, F32)
    keys = np.zeros((U, 7), np.uint64)
    reach = np.full((U, 7), -1, np.int64)
    cur = np.zeros(U, np.int64)
    curc = C[:, 0].copy()
    prev = np.full(U, np.inf, F32)
    alive = np.ones(U, bool)
    low = (np.uint64(0xFFFFFFFF) - np.arange(U, dtype=np.uint64))
    with np.errstate(divide="ignore", invalid="ignore"):
        for step in range(7):
            best_e = np.zeros(U, F32)
            best_j = np.full(U, -1, np.int64)
            for j in range(1, 8):
                db = bits[j] - bits[cur]
                e = (curc - C[:, j]) / db
                ok = alive & (j > cur) & (e > 0) & (e > best_e)
                best_e = np.where(ok, e, best_e)
                best_j = np.where(ok, j, best_j)
            has = best_j >= 0
            e = np.minimum(best_e, prev)
            kb = e.view(np.uint32).astype(np.uint64)
            keys[:, step] = np.where(has, (kb << np.uint64(32)) | low, np.uint64(0))
            reach[:, step] = np.where(has, best_j, -1)
            nj = np.where(has, best_j, 0)
            curc = np.where(has, C[np.arange(U), nj], curc)
            cur = np.where(has, best_j, cur)
            prev = np.where(has, e, prev)
            alive &= has
    return keys, reach


def allocate(C: np.ndarray, budget: int, fill: bool = True) -> np.ndarray:
    """Bit-width per unit (uint8) by steps 2-4 for the cost table C (U x 8, fp32);
    fill=False stops after step 3 (the Lagrangian solution)."""
    keys, reach = hull_increments(C)
    U = keys.shape[0]
    bits = np.array(BITS, np.int64)
    # step deltas in bits
    prev_b = np.concatenate([np.zeros((U, 1), np.int64), np.where(reach >= 0, bits[np.maximum(reach, 0)], 0)[:, :-1]],
                            axis=1)
    db = np.where(reach >= 0, bits[np.maximum(reach, 0)] - prev_b, 0)
    flat = keys.reshape(-1)
    live = flat > 0
    kk, dd = flat[live], db.reshape(-1)[live]
    order = np.argsort(kk, kind="stable")[::-1]          # descending keys
    kk, dd = kk[order], dd[order]
    csum = np.cumsum(dd)
    # groups of equal keys are taken whole: the cut is the first key whose group overflows
    if csum.size and csum[-1] > budget:
        first_over = int(np.argmax(csum > budget))
        kstar = kk[first_over]
    else:
        kstar = np.uint64(0)
    taken = (keys > kstar).sum(axis=1)                   # prefix lengths (keys never increase)
    used = int(np.where(taken > 0, db.cumsum(axis=1)[np.arange(U), np.maximum(taken - 1, 0)], 0).sum())
    R = budget - used
    # step 4: greedy fill with each unit's next increment
    while fill:
        nxt = np.where(taken < 7, taken, 6)
        cand_key = np.where(taken < 7, keys[np.arange(U), nxt], np.uint64(0))
        cand_db = np.where(taken < 7, db[np.arange(U), nxt], 0)
        ok = (cand_key > 0) & (cand_db <= R)
        if not ok.any():
            break
        u = int(np.argmax(np.where(ok, cand_key, np.uint64(0))))
        R -= int(cand_db[u])
        taken[u] += 1
    out = np.zeros(U, np.uint8)
    has = taken > 0
    out[has] = bits[reach[np.arange(U), np.maximum(taken - 1, 0)][has]]
    return out


def total_cost(C: np.ndarray, b: np.ndarray) -> float:
    """sum_u C_u(b_u) in fp64."""
    idx = np.searchsorted(np.array(BITS), np.asarray(b, np.int64))
    return float(np.asarray(C, np.float64)[np.arange(len(idx)), idx].sum())


def ilp_optimum(C: np.ndarray, budget: int) -> Tuple[float, np.ndarray]:
    """Exact optimum of Eq. ilp_piecewise_eps by dynamic programming over the budget (fp64;
    tiny inputs only): returns (cost, bits)."""
    C = np.asarray(C, np.float64)
    U = C.shape[0]
    INF = float("inf")
    best = np.full(budget + 1, INF)
    best[0] = 0.0
    choice = np.zeros((U, budget + 1), np.int64)
    for u in range(U):
        nb = np.full(budget + 1, INF)
        for j, b in enumerate(BITS):
            if b > budget:
                continue
            cand = np.full(budget + 1, INF)
            cand[b:] = best[:budget + 1 - b] + C[u, j]
            better = cand < nb
            nb = np.where(better, cand, nb)
            choice[u] = np.where(better, j, choice[u])
        best = nb
    B = int(np.argmin(best))
    cost = float(best[B])
    out = np.zeros(U, np.uint8)
    for u in range(U - 1, -1, -1):
        j = int(choice[u, B])
        out[u] = BITS[j]
        B -= BITS[j]
    return cost, out


def lp_bound(C: np.ndarray, budget: int) -> float:
    """Value of the LP relaxation at the budget (a lower bound on the ILP optimum): the
    hull increments taken in descending efficiency, the last one fractionally (fp64)."""
    C = np.asarray(C, np.float64)
    U = C.shape[0]
    incs = []
    base = float(C[:, 0].sum())
    for u in range(U):
        cur = 0
        while True:
            best, bj = 0.0, -1
            for j in range(cur + 1, 8):
                e = (C[u, cur] - C[u, j]) / (BITS[j] - BITS[cur])
                if e > 0 and e > best:
                    best, bj = e, j
            if bj < 0:
                break
            incs.append((best, BITS[bj] - BITS[cur], C[u, cur] - C[u, bj]))
            cur = bj
    incs.sort(key=lambda t: -t[0])
    left, val = float(budget), base
    for e, db, gain in incs:
        if db <= left:
            val -= gain
            left -= db
        else:
            val -= gain * left / db
            break
    return val
