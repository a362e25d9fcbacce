"""fp64 CPU oracle for the BitsMoE quantized MoE-layer forward (Stage 3).

TEST INFRASTRUCTURE ONLY.  This is the plain, slow, obviously correct statement
of what the GPU path computes, used to check it.  Only ``tests/``,
``__graft_entry__.smoke()`` and the ``cpu_baseline`` / ``--impl reference``
legs of ``bench.py`` may import it.  It shares no code with the CUDA library
and imports nothing from it; inputs come from the seeded generator ``synth``.

Passages followed (BitsMoE paper):
* Shared-basis decomposition, Sec. "Shared-basis Spectral Decomposition"
  (Eq. shared_basis_input_proj for gate/up, the down_proj concatenation along
  the input channels) and its appendix restatement (Eqs. app_w_cat ...
  app_down_p_tilde_partition).
* Spectral energy alpha and the normalised spectral matrix P
  (Definitions spectral_energy_matrix / spectral_matrix,
  Eq. app_normalized_decomposition):
      W_e = P_e A_e Phi^T  (gate, up),     W_e = Phi A_e P_e^T  (down).
* Quantisation acts on the normalised spectral vectors only, and the quantised
  weight is W_hat = P_hat A Phi^T (Eqs. quantized_spectral_vector and
  reconstruction_error_compact); the basis stays unquantised.
* Per-unit quantisers: symmetric uniform Q_b (Eq. app_scalar_quantization_uk,
  MSE-optimal scale of Eq. app_lowbit_empirical_error), the 1-bit sign
  quantiser with sign(0) = +1 (Eq. app_one_bit_quantization) and 0-bit
  eviction Q_0 = 0 (Eq. app_zero_bit_vector).  Group size 128 in the paper's
  experiments (Sec. Experimental Setup, Baselines).
* Stage 3 of Fig. 1 (overview): inputs are projected onto the shared basis and
  the quantised spectral factors compute the routed experts; SwiGLU
  gate/up/down projections (Sec. Shared-basis Spectral Decomposition).

Readings where the paper is silent (the same readings on the CUDA side):
* stored format of a unit of b bits, 0 < b < 16: unsigned codes q in
  [0, 2^b) with one fp16 scale s and fp16 zero z per group of `group`
  consecutive elements along the unit vector, p_hat[i] = s[g(i)] * (q[i] - z[g(i)]).
  The paper's symmetric quantiser is the case z = 2^(b-1); its 1-bit sign
  quantiser is the case z = 1/2, s = 2 * mean|p|.
* b = 16: the unit is stored as fp16 values, no scale or zero.
* routing: the k largest logits (ties go to the lower expert index), gate
  weights = softmax over the selected k logits.
* SwiGLU: h = SiLU(gate) * up, SiLU(a) = a / (1 + exp(-a)).
"""
from __future__ import annotations

import math
from typing import Dict, List, Sequence, Tuple

import numpy as np

GATE, UP, DOWN = 0, 1, 2


# ----------------------------------------------------------------------------
# Stored values -> exact fp64
# ----------------------------------------------------------------------------
def bf16_bits_to_f64(u16: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> their exact values."""
    u = np.asarray(u16, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def f16_bits_to_f64(u16: np.ndarray) -> np.ndarray:
    """fp16 bit patterns -> their exact values."""
    return np.asarray(u16, dtype=np.uint16).view(np.float16).astype(np.float64)


# ----------------------------------------------------------------------------
# Dequantisation of one spectral unit and of a whole expert factor P_hat
# ----------------------------------------------------------------------------
def dequantize_unit(b: int, codes: np.ndarray, scale: np.ndarray, zero: np.ndarray,
                    group: int) -> np.ndarray:
    """p_hat for one unit of length I (the quantised spectral vector).

    b = 0: the unit is evicted, p_hat = 0 (Eq. app_zero_bit_vector).
    b = 16: fp16 values as stored.
    otherwise: p_hat[i] = s[g] * (q[i] - z[g]) with g = i // group.
    """
    I = codes.shape[-1]
    if b == 0:
        return np.zeros(I, dtype=np.float64)
    if b == 16:
        return f16_bits_to_f64(codes)
    g = np.arange(I) // group
    s = f16_bits_to_f64(scale)[g]
    z = f16_bits_to_f64(zero)[g]
    return s * (codes.astype(np.float64) - z)


def dequantize_factor(layer: Dict, h: int, e: int) -> np.ndarray:
    """P_hat_e^(h) as an I x n matrix whose column k is p_hat_{e,h,k}: the
    per-unit definition of dequantize_unit applied to all units at once."""
    I, n, group = layer["I"], layer["n"], layer["group"]
    bits = np.asarray(layer["bits"][h, e])
    codes = layer["codes"][h, e]
    P = np.zeros((n, I), dtype=np.float64)          # row k = unit k
    q = (bits > 0) & (bits < 16)
    if q.any():
        g = np.arange(I) // group
        s = f16_bits_to_f64(layer["scale"][h, e][q])[:, g]
        z = f16_bits_to_f64(layer["zero"][h, e][q])[:, g]
        P[q] = s * (codes[q].astype(np.float64) - z)
    f = bits == 16
    if f.any():
        P[f] = f16_bits_to_f64(codes[f])
    return P.T


def basis(layer: Dict, h: int) -> np.ndarray:
    """Phi_h (D x n) in fp64."""
    return bf16_bits_to_f64(layer["basis"][h])


def alpha(layer: Dict, h: int, e: int) -> np.ndarray:
    return np.asarray(layer["alpha"][h, e], dtype=np.float64)


# ----------------------------------------------------------------------------
# Dense (definition) form: W_hat_e = P_hat A Phi^T (gate/up), Phi A P_hat^T (down)
# ----------------------------------------------------------------------------
def expert_weights(layer: Dict, e: int) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """Quantised expert weights (W_gate I x D, W_up I x D, W_down D x I)."""
    out = []
    for h in (GATE, UP):
        P = dequantize_factor(layer, h, e)
        out.append(P @ np.diag(alpha(layer, h, e)) @ basis(layer, h).T)
    P = dequantize_factor(layer, DOWN, e)
    out.append(basis(layer, DOWN) @ np.diag(alpha(layer, DOWN, e)) @ P.T)
    return out[0], out[1], out[2]


def silu(a: np.ndarray) -> np.ndarray:
    return a / (1.0 + np.exp(-a))


def route(logits: np.ndarray, top_k: int) -> Tuple[np.ndarray, np.ndarray]:
    """Top-k experts per token (largest logit first, ties to the lower index)
    and their gate weights, a softmax over the k selected logits."""
    logits = np.asarray(logits, dtype=np.float64)
    T, E = logits.shape
    idx = np.empty((T, top_k), dtype=np.int64)
    w = np.empty((T, top_k), dtype=np.float64)
    for t in range(T):
        order = np.lexsort((np.arange(E), -logits[t]))[:top_k]
        sel = logits[t, order]
        ex = np.exp(sel - sel.max())
        idx[t] = order
        w[t] = ex / ex.sum()
    return idx, w


def moe_forward_dense(layer: Dict, x_bits: np.ndarray, logits: np.ndarray,
                      top_k: int) -> np.ndarray:
    """y_t = sum_{e in topk(t)} g_{t,e} W_dn,e (SiLU(W_g,e x_t) * W_u,e x_t), fp64."""
    x = bf16_bits_to_f64(x_bits)
    idx, w = route(logits, top_k)
    T = x.shape[0]
    y = np.zeros((T, layer["D"]), dtype=np.float64)
    cache = {}
    for t in range(T):
        for s in range(top_k):
            e = int(idx[t, s])
            if e not in cache:
                cache[e] = expert_weights(layer, e)
            Wg, Wu, Wd = cache[e]
            y[t] += w[t, s] * (Wd @ (silu(Wg @ x[t]) * (Wu @ x[t])))
    return y


# ----------------------------------------------------------------------------
# Factored form (Stage 3): project once on the shared basis, then the factors
# ----------------------------------------------------------------------------
def moe_forward_factored(layer: Dict, x_bits: np.ndarray, logits: np.ndarray,
                         top_k: int, return_parts: bool = False):
    """Same map as moe_forward_dense, associated as the paper's inference path:
    z_h = Phi_h^T x (once per layer), gate = P_hat_g (alpha_g * z_g),
    up = P_hat_u (alpha_u * z_u), h = SiLU(gate) * up,
    s = sum_e g_e alpha_dn,e * (P_hat_dn,e^T h_e), y = Phi_dn s."""
    x = bf16_bits_to_f64(x_bits)
    idx, w = route(logits, top_k)
    T = x.shape[0]
    zg = x @ basis(layer, GATE)          # T x n, row t = Phi_g^T x_t
    zu = x @ basis(layer, UP)
    s_acc = np.zeros((T, layer["n"]), dtype=np.float64)
    hidden = {}
    for e in sorted(set(int(v) for v in idx.ravel())):   # one expert's factors at a time
        Pg, Pu, Pd = (dequantize_factor(layer, h, e) for h in (GATE, UP, DOWN))
        for t, s in zip(*np.nonzero(idx == e)):
            gate = Pg @ (alpha(layer, GATE, e) * zg[t])
            up = Pu @ (alpha(layer, UP, e) * zu[t])
            hvec = silu(gate) * up
            hidden[(int(t), e)] = hvec
            s_acc[t] += w[t, s] * alpha(layer, DOWN, e) * (Pd.T @ hvec)
        del Pg, Pu, Pd
    y = s_acc @ basis(layer, DOWN).T
    if return_parts:
        return y, dict(idx=idx, w=w, zg=zg, zu=zu, s=s_acc, hidden=hidden)
    return y


def moe_forward_factored_token(layer: Dict, x_bits_row: np.ndarray, logits_row: np.ndarray,
                               top_k: int, cache: Dict = None) -> np.ndarray:
    """One token of moe_forward_factored (for sampled checks at full size)."""
    return moe_forward_factored(layer, x_bits_row[None, :], logits_row[None, :], top_k)[0]


# ----------------------------------------------------------------------------
# Layer stack (pre-norm residual MoE FFN blocks)
# ----------------------------------------------------------------------------
def rms_norm(h: np.ndarray, eps: float = 1e-6) -> np.ndarray:
    """RMSNorm with unit weight: h / sqrt(mean(h^2) + eps), per row."""
    h = np.asarray(h, dtype=np.float64)
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps)


def router_logits(w_router_bits: np.ndarray, x_bits: np.ndarray) -> np.ndarray:
    """Router logits W_r x of a stacked MoE block (W_r: E x D bf16 bits, x: T x D bf16 bits)."""
    return bf16_bits_to_f64(x_bits) @ bf16_bits_to_f64(w_router_bits).T


# ----------------------------------------------------------------------------
# Offline pieces used by the pins (not on the hot path)
# ----------------------------------------------------------------------------
def shared_basis_decompose(W: Sequence[np.ndarray], side: str):
    """Shared-basis decomposition of one projection type over E experts.

    side == "in"  (gate/up): W_cat = [W_1; ...; W_E] = U S Phi^T, P~_cat = U S
                             split into E row blocks (Eq. app_cat_svd_absorbed).
    side == "out" (down):    W_cat = [W_1 ... W_E] = Phi S V^T, P~_cat = V S
                             split by input-channel blocks (Eq. app_down_cat_svd_absorbed).
    Then alpha_{e,k} = ||p~_{e,k}||_2 and P_e = P~_e A_e^{-1}
    (Definitions spectral_energy_matrix / spectral_matrix).
    Returns Phi (feature dim x n), alpha (E x n), P (list of E arrays, d x n).
    """
    W = [np.asarray(w, dtype=np.float64) for w in W]
    if side == "in":
        Wcat = np.concatenate(W, axis=0)
        U, S, Vt = np.linalg.svd(Wcat, full_matrices=False)
        Phi = Vt.T
        Pcat = U * S[None, :]
        rows = [w.shape[0] for w in W]
    elif side == "out":
        Wcat = np.concatenate(W, axis=1)
        U, S, Vt = np.linalg.svd(Wcat, full_matrices=False)
        Phi = U
        Pcat = Vt.T * S[None, :]
        rows = [w.shape[1] for w in W]
    else:
        raise ValueError(side)
    blocks = np.split(Pcat, np.cumsum(rows)[:-1], axis=0)
    alphas = np.stack([np.linalg.norm(b, axis=0) for b in blocks])
    P = [b / np.where(a > 0, a, 1.0)[None, :] for b, a in zip(blocks, alphas)]
    return Phi, alphas, P


def quantize_symmetric(p: np.ndarray, b: int, s: float) -> np.ndarray:
    """Integer levels of the symmetric uniform quantiser,
    clamp(round(p / s), -2^(b-1), 2^(b-1) - 1) (Eq. app_scalar_quantization_uk).
    round() is round-half-to-even."""
    qmin, qmax = -(1 << (b - 1)), (1 << (b - 1)) - 1
    return np.clip(np.rint(np.asarray(p, dtype=np.float64) / s), qmin, qmax).astype(np.int64)


def mse_optimal_scale(p: np.ndarray, b: int, grid: int = 400) -> float:
    """s* = argmin_s ||p - Q_b(p; s)||^2 by a dense search over
    s in (0, max|p| / 2^(b-2)] (Eq. app_lowbit_empirical_error)."""
    p = np.asarray(p, dtype=np.float64)
    top = np.max(np.abs(p)) / max(1 << (b - 1), 1) * 2.0
    cands = top * np.arange(1, grid + 1) / grid
    best, best_err = cands[-1], np.inf
    for s in cands:
        err = np.sum((p - s * quantize_symmetric(p, b, s)) ** 2)
        if err < best_err:
            best, best_err = s, err
    return float(best)


def quantize_sign(p: np.ndarray) -> Tuple[np.ndarray, float]:
    """1-bit sign quantiser: signs (sign(0) = +1) and s_1 = mean|p|
    (Eq. app_one_bit_quantization)."""
    p = np.asarray(p, dtype=np.float64)
    sg = np.where(p >= 0, 1, -1).astype(np.int64)
    return sg, float(np.mean(np.abs(p)))
