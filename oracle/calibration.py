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

Reading (the paper does not fix it): a token's routing affinity to expert e is its gate weight
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


def swiglu_intermediate(Phi_g: np.ndarray, Phi_u: np.ndarray, Pa_g: np.ndarray, Pa_u: np.ndarray,
                        X: np.ndarray) -> np.ndarray:
    """h = SiLU(P_g A_g Phi_g^T X) * (P_u A_u Phi_u^T X) (I x T) for activations X (D x T),
    given the factors with their energies folded in (Pa = P diag(alpha), I x n)."""
    gate = Pa_g @ (np.asarray(Phi_g, np.float64).T @ X)
    up = Pa_u @ (np.asarray(Phi_u, np.float64).T @ X)
    return silu(gate) * up


def intermediate(layer, x_bits: np.ndarray, e: int) -> np.ndarray:
    """The expert's SwiGLU output h = SiLU(W_gate x) * (W_up x) for every token (I x T) with
    the stored (quantised) factors: the activations entering its down projection."""
    X = bf16_bits_to_f64(x_bits).T                                   # D x T
    Pa_g = dequantize_factor(layer, GATE, e) * alpha(layer, GATE, e)[None, :]
    Pa_u = dequantize_factor(layer, UP, e) * alpha(layer, UP, e)[None, :]
    return swiglu_intermediate(basis(layer, GATE), basis(layer, UP), Pa_g, Pa_u, X)


def factor_importance(Phi, alpha_, P, x_bits: np.ndarray, logits: np.ndarray, top_k: int) -> np.ndarray:
    """beta[h][e, k] from the decomposition's float factors, before any quantisation.

    Phi[h]: D x n bases (h = gate, up, down); alpha_[h]: E x n energies; P[h][e]: I x n
    normalised spectral factors.  This is the allocation's input: the importance weights the
    loss of quantising each unit (appendix Eq. app_unified_beta_def), so it is taken on the
    unquantised factors, and the down projection's activations are the expert's SwiGLU
    outputs of the float layer (appendix Eq. app_down_beta_approx).
    """
    E, n = np.asarray(alpha_[0]).shape
    g = affinities(logits, top_k, E)
    X = bf16_bits_to_f64(x_bits).T
    out = np.zeros((3, E, n))
    for e in range(E):
        H_in = activation_metric(X, g[:, e])
        out[GATE, e] = importance(Phi[GATE], H_in)
        out[UP, e] = importance(Phi[UP], H_in)
        Pa_g = np.asarray(P[GATE][e], np.float64) * np.asarray(alpha_[GATE][e], np.float64)[None, :]
        Pa_u = np.asarray(P[UP][e], np.float64) * np.asarray(alpha_[UP][e], np.float64)[None, :]
        H_dn = activation_metric(swiglu_intermediate(Phi[GATE], Phi[UP], Pa_g, Pa_u, X), g[:, e])
        out[DOWN, e] = importance(np.asarray(P[DOWN][e], np.float64), H_dn)
    return out


def layer_importance(layer, x_bits: np.ndarray, logits: np.ndarray, top_k: int) -> Tuple[np.ndarray, ...]:
    """beta[h][e, k] of a stored (quantised) layer on calibration tokens (x, logits): the same
    definition as factor_importance with the dequantised factors in place of the float ones.
    Used by the eviction-loss pin, whose loss is measured on the stored layer."""
    E = int(layer["E"])
    Phi = [basis(layer, h) for h in (GATE, UP, DOWN)]
    al = [np.stack([alpha(layer, h, e) for e in range(E)]) for h in (GATE, UP, DOWN)]
    P = [[dequantize_factor(layer, h, e) for e in range(E)] for h in (GATE, UP, DOWN)]
    return factor_importance(Phi, al, P, x_bits, logits, top_k)
