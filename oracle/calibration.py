"""CPU oracle of the activation-aware importance beta (calibration side of the allocation).

TEST INFRASTRUCTURE ONLY, like the rest of ``oracle/``: imported by tests/ only, never by
the CUDA library or its binding, and it shares no code with them.  fp64 throughout.

What the paper defines (Sec. "Shared-basis Spectral Decomposition", the reconstruction
loss lemma; appendix Eqs. app_beta_def, app_down_beta_approx, app_unified_beta_def):

* the activation metric of one expert and projection, H = X Diag(g) X^T, where the
  columns of X are the calibration activations entering the projection and g weights each
  by its routing affinity to the expert;
* beta_k = phi_k^T H phi_k for the gate and up projections (the shared input basis), and
  beta_k = p_k^T H p_k for the down projection (the expert-specific vector, H over the
  expert's intermediate activations).

Reading (listed in the design doc): a token's routing affinity to expert e is its gate weight
(the softmax over its k selected experts) when e is selected and 0 otherwise, the same
weights the forward applies.
"""
from __future__ import annotations

from typing import Tuple

import numpy as np

from .bitsmoe_oracle import (DOWN, GATE, UP, alpha, basis, bf16_bits_to_f64, dequantize_factor, route,
                             silu)


def activation_metric(X: np.ndarray, g: np.ndarray) -> np.ndarray:
    """H = X Diag(g) X^T for activations X (features x tokens) and token weights g."""
    X = np.asarray(X, np.float64)
    return (X * np.asarray(g, np.float64)[None, :]) @ X.T


def importance(V: np.ndarray, H: np.ndarray) -> np.ndarray:
    """beta_k = v_k^T H v_k for the columns v_k of V (Eq. app_unified_beta_def)."""
    V = np.asarray(V, np.float64)
    return np.einsum("ik,ij,jk->k", V, np.asarray(H, np.float64), V)


def affinities(logits: np.ndarray, top_k: int, E: int) -> np.ndarray:
    """g[t, e]: gate weight of expert e for token t if selected, else 0 (T x E)."""
    idx, w = route(logits, top_k)
    g = np.zeros((idx.shape[0], E))
    for t in range(idx.shape[0]):
        g[t, idx[t]] = w[t]
    return g


def intermediate(layer, x_bits: np.ndarray, e: int) -> np.ndarray:
    """The expert's SwiGLU output h = SiLU(W_gate x) * (W_up x) for every token (I x T):
    the activations entering its down projection."""
    X = bf16_bits_to_f64(x_bits).T                                   # D x T
    zg = basis(layer, GATE).T @ X
    zu = basis(layer, UP).T @ X
    a_g = alpha(layer, GATE, e)[:, None]
    a_u = alpha(layer, UP, e)[:, None]
    gate = dequantize_factor(layer, GATE, e) @ (a_g * zg)
    up = dequantize_factor(layer, UP, e) @ (a_u * zu)
    return silu(gate) * up


def layer_importance(layer, x_bits: np.ndarray, logits: np.ndarray, top_k: int) -> Tuple[np.ndarray, ...]:
    """beta[h][e, k] of every projection and expert on calibration tokens (x, logits)."""
    E, n = int(layer["E"]), int(layer["n"])
    g = affinities(logits, top_k, E)
    X = bf16_bits_to_f64(x_bits).T
    out = np.zeros((3, E, n))
    for e in range(E):
        H_in = activation_metric(X, g[:, e])
        out[GATE, e] = importance(basis(layer, GATE), H_in)
        out[UP, e] = importance(basis(layer, UP), H_in)
        H_dn = activation_metric(intermediate(layer, x_bits, e), g[:, e])
        out[DOWN, e] = importance(dequantize_factor(layer, DOWN, e), H_dn)
    return out
