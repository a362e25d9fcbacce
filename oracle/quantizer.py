"""CPU oracle of the per-unit quantiser (normalised spectral vectors -> stored units).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: imported by tests/ and
by the CPU legs of bench.py, never by the CUDA library or its binding, and it
shares no code with them.

What it computes (BitsMoE paper, appendix "Piecewise Reconstruction Error for
Bit Allocation"): each spectral unit p (a column of P, length I) is quantised
with its own bit-width b in {0, 1, 2, 3, 4, 6, 8, 16}, one scale per group of
``group`` consecutive elements (group size 128 in Sec. Experimental Setup):

* b in {2, 3, 4}: the symmetric uniform quantiser of Eq.
  app_scalar_quantization_uk, Q_b(p; s) = s * clamp(round(p / s), -2^(b-1),
  2^(b-1) - 1), with the MSE-optimal scale of Eq. app_low_bit_opt_scale,
  s* = argmin_s ||p - Q_b(p; s)||^2, searched over `grid` candidates;
* b in {6, 8}: the same quantiser with s = rho / q_max, rho = ||p||_inf
  (Eqs. app_high_bit_rho_eta and app_uk_scale);
* b = 1: the sign quantiser of Eq. app_one_bit_quantization, s_1 * sign(p) with
  s_1 = mean |p| and sign(0) = +1;
* b = 0: the unit is evicted (Eq. app_zero_bit_vector);
* b = 16: the unit is kept as fp16 values.

Stored format (the one the forward reads): unsigned codes, fp16 scale and zero
per group, p_hat = scale * (code - zero).  Symmetric levels q are stored as
code = q + 2^(b-1) with zero = 2^(b-1); the sign quantiser as code = [p >= 0],
zero = 1/2, scale = 2 s_1.

Readings where the paper leaves the arithmetic open:
* precision: fp32, every operation rounded once to nearest-even (no fused
  multiply-add in the error sums); the quotient p / s is taken as p times the
  fp32 reciprocal of s (within one ulp of the quotient: a code exactly at a
  half-way point may differ by one from an exact division, at equal error);
* candidate scales: s_c = fp16(fp32(top * c) / grid), c = 1 .. grid, top =
  rho * 2^(2-b) (twice the scale that maps rho to 2^(b-1)), so every candidate
  is a storable scale; scales that are 0 or not finite in fp16 are skipped;
* the squared error of a candidate is summed over the group's elements in
  order; the smallest error wins, ties to the smaller candidate index c;
* a group with no usable scale (rho = 0, or every candidate skipped; for
  b in {6, 8} a scale of 0 or infinity) stores scale 0 and the zero level;
* b = 1: mean |p| is summed over the group's elements in order and divided by
  the group size; its scale 2 s_1 is rounded to fp16.
"""
from __future__ import annotations

from typing import Tuple

import numpy as np

SUPPORTED_BITS = (0, 1, 2, 3, 4, 6, 8, 16)
F32 = np.float32


def _f16(a: np.ndarray) -> np.ndarray:
    """Round fp32 values to fp16 (nearest-even) and back to fp32."""
    return np.asarray(a, dtype=F32).astype(np.float16).astype(F32)


def _f16_bits(a: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=F32).astype(np.float16)).view(np.uint16)


def _levels(X: np.ndarray, s: np.ndarray, b: int) -> np.ndarray:
    """q = clamp(round(p / s), q_min, q_max) per element, the quotient as p * fp32(1 / s).
    X: (..., g) fp32 values, s: (...) or broadcastable fp32 scales (> 0)."""
    qmin, qmax = F32(-(1 << (b - 1))), F32((1 << (b - 1)) - 1)
    with np.errstate(divide="ignore", invalid="ignore", over="ignore"):
        r = F32(1.0) / np.asarray(s, dtype=F32)
        return np.rint(np.clip(X * r, qmin, qmax))


def _usable(s: np.ndarray) -> np.ndarray:
    return (s > 0) & np.isfinite(s)


def _mse_search(X: np.ndarray, b: int, grid: int) -> np.ndarray:
    """MSE-optimal fp16 scale per group (rows of X), Eq. app_low_bit_opt_scale over the
    candidate set; 0 where no candidate is usable."""
    G, g = X.shape
    rho = np.max(np.abs(X), axis=1)                                   # ||p||_inf per group
    top = rho * F32(2.0 ** (2 - b))                                   # exact power-of-two scaling
    c = np.arange(1, grid + 1, dtype=F32)
    with np.errstate(over="ignore"):
        S = _f16((top[:, None] * c[None, :]) / F32(grid))             # G x grid candidates
    ok = _usable(S)
    Sx = np.where(ok, S, F32(1.0))                                    # placeholder for skipped ones
    err = np.zeros((G, grid), dtype=F32)
    qmin, qmax = F32(-(1 << (b - 1))), F32((1 << (b - 1)) - 1)
    R = F32(1.0) / Sx
    with np.errstate(over="ignore", invalid="ignore"):
        for i in range(g):                                            # elements in order
            v = X[:, i][:, None]
            q = np.rint(np.clip(v * R, qmin, qmax))
            d = v - Sx * q                                            # Sx * q is exact in fp32
            err = err + d * d
    err = np.where(ok, err, F32(np.inf))
    best = np.argmin(err, axis=1)                                     # first minimum: smallest c
    s = S[np.arange(G), best]
    none = ~np.isfinite(err[np.arange(G), best])
    return np.where(none, F32(0.0), s).astype(F32)


def _sign_scale(X: np.ndarray) -> np.ndarray:
    """2 * s_1 per group, s_1 = mean |p| (Eq. app_one_bit_quantization), fp16-rounded."""
    G, g = X.shape
    acc = np.zeros(G, dtype=F32)
    for i in range(g):
        acc = acc + np.abs(X[:, i])
    return _f16(F32(2.0) * (acc / F32(g)))


def quantize_units(P: np.ndarray, bits: np.ndarray, group: int, grid: int = 256
                   ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Quantise U units (rows of P, each of length I) into the stored format.

    P: U x I float32 (finite), bits: U bit-widths in SUPPORTED_BITS, I % group == 0.
    Returns codes (U x I uint16), scale and zero (U x I/group fp16 bit patterns).
    """
    P = np.ascontiguousarray(P, dtype=F32)
    bits = np.asarray(bits).reshape(-1)
    U, I = P.shape
    if bits.size != U or I % group:
        raise ValueError("shape")
    if not set(np.unique(bits).tolist()) <= set(SUPPORTED_BITS):
        raise ValueError("unsupported bit-width")
    ng = I // group
    codes = np.zeros((U, I), np.uint16)
    scale = np.zeros((U, ng), np.uint16)
    zero = np.zeros((U, ng), np.uint16)
    for b in np.unique(bits).tolist():
        rows = np.nonzero(bits == b)[0]
        if b == 0 or rows.size == 0:
            continue
        X = P[rows].reshape(-1, group)                                # one row per (unit, group)
        if b == 16:
            codes[rows] = _f16_bits(P[rows])
            continue
        if b == 1:
            s2 = _sign_scale(X)
            q = (X >= 0).astype(np.uint16)
            z = np.full(X.shape[0], 0.5, F32)
        else:
            half = F32(1 << (b - 1))
            if b in (2, 3, 4):
                s2 = _mse_search(X, b, grid)
            else:
                rho = np.max(np.abs(X), axis=1)
                with np.errstate(over="ignore"):
                    s2 = _f16(rho / F32((1 << (b - 1)) - 1))
                s2 = np.where(_usable(s2), s2, F32(0.0)).astype(F32)
            ok = _usable(s2)
            lv = _levels(X, np.where(ok, s2, F32(1.0))[:, None], b)
            lv = np.where(ok[:, None], lv, F32(0.0))
            q = (lv + half).astype(np.uint16)
            z = np.full(X.shape[0], half, F32)
        codes[rows] = q.reshape(rows.size, I)
        scale[rows] = _f16_bits(s2).reshape(rows.size, ng)
        zero[rows] = _f16_bits(z).reshape(rows.size, ng)
    return codes, scale, zero

