"""Seeded synthetic BitsMoE layers and decode inputs.

This module is the one piece shared by the CUDA path's tests/benchmark and the
fp64 oracle: it only draws random numbers and stores them in the storage
formats both sides read (bf16 / fp16 bit patterns, integer codes, fp32).  It
holds none of the method's arithmetic (no dequantisation, no projection, no
routing).

Workloads are the shapes of the paper's evaluated MoE layers (Qwen3-30B-A3B,
Mixtral-8x7B, plus a tiny layer); no model weights or datasets are used.
Recipe (one ``numpy.random.Generator`` per layer, draws in this order):

1. three shared bases Phi_h (h = gate, up, down), each the Q factor of a QR
   decomposition of an N(0, 1/D) D x n matrix, rounded to bf16 (layers of the
   48-layer stack instead use a random signed permutation times two random
   Householder reflections: also orthonormal, dense, and cheap enough to draw
   48 layers);
2. per-unit bit-widths b[h, e, j] i.i.d. from the config's distribution;
3. integer codes uniform on [0, 2^b) for every element of every unit: the low
   b bits of 4-bit (blocks whose units have at most 4 bits) or 16-bit fields
   cut from SplitMix64 outputs (Steele, Lea, Flood 2014) of the counter
   key(seed, layer) + i, computed block by block in threads
   (b = 16 units instead hold fp16 values drawn N(0, 1/I) from the layer generator);
4. per (unit, group) fp16 scale 2*sqrt(3/I)/(2^b - 1) * U(0.75, 1.25) and fp16
   zero (2^b - 1)/2 + U(-0.5, 0.5) (so dequantised units have about unit norm,
   like the paper's normalised spectral vectors, while every group differs);
5. spectral energies alpha[h, e, j] = alpha_scale * j^(-1/2) (fp32).

Decode inputs come from a separate generator per (seed, step, T): activations
x ~ N(0, 1) rounded to bf16 and router logits ~ N(0, 1) in fp32, plus a fixed
per-expert bias drawn N(0, std) for the skewed-load workload.
"""
from __future__ import annotations

import dataclasses
import math
import os
from concurrent.futures import ThreadPoolExecutor
from typing import Dict, Optional, Sequence, Tuple

import numpy as np

# Candidate bit-widths of the paper's allocation (0 = evicted unit, 16 = fp16 unit).
BIT_CANDIDATES = (0, 1, 2, 3, 4, 6, 8, 16)

DIST_MEAN_2_0 = {0: 0.1, 1: 0.2, 2: 0.4, 3: 0.2, 4: 0.1}
DIST_MEAN_2_5 = {1: 0.1, 2: 0.4, 3: 0.4, 4: 0.1}

GATE, UP, DOWN = 0, 1, 2


@dataclasses.dataclass(frozen=True)
class LayerSpec:
    name: str
    D: int          # hidden size
    E: int          # routed experts
    I: int          # expert intermediate size (length of a spectral unit)
    n: int          # shared-basis rank (units per expert and projection)
    group: int      # quantisation group along the unit vector
    top_k: int
    bits_dist: Tuple[Tuple[int, float], ...]
    tokens: Tuple[int, ...]
    expert_bias_std: float = 0.0
    layers: int = 1

    @property
    def mean_bits(self) -> float:
        return float(sum(b * p for b, p in self.bits_dist))


def _dist(d: Dict[int, float]) -> Tuple[Tuple[int, float], ...]:
    return tuple(sorted(d.items()))


WORKLOADS: Dict[str, LayerSpec] = {
    # tiny layer: parity case the oracle finishes in well under a second
    "tiny": LayerSpec("tiny", D=256, E=8, I=512, n=256, group=64, top_k=2,
                      bits_dist=_dist(DIST_MEAN_2_0), tokens=(4,)),
    # Qwen3-30B-A3B-shaped MoE layer, batch-1 decode at 2.0 mean unit bits
    "qw3": LayerSpec("qw3", D=2048, E=128, I=768, n=2048, group=128, top_k=8,
                     bits_dist=_dist(DIST_MEAN_2_0), tokens=(1,)),
    # same shape, 2.5 mean bits, skewed expert load, decode batch 1/8/32/128
    "qw3_skew": LayerSpec("qw3_skew", D=2048, E=128, I=768, n=2048, group=128, top_k=8,
                          bits_dist=_dist(DIST_MEAN_2_5), tokens=(1, 8, 32, 128),
                          expert_bias_std=1.5),
    # Mixtral-8x7B-shaped MoE layer, decode batch 1 and 16
    "mixtral": LayerSpec("mixtral", D=4096, E=8, I=14336, n=4096, group=128, top_k=2,
                         bits_dist=_dist(DIST_MEAN_2_0), tokens=(1, 16)),
    # 48-layer Qwen3-30B-A3B-shaped MoE FFN stack (RMSNorm between layers)
    "qw3_stack": LayerSpec("qw3_stack", D=2048, E=128, I=768, n=2048, group=128, top_k=8,
                           bits_dist=_dist(DIST_MEAN_2_0), tokens=(1, 32), layers=48),
}


def scaled_spec(spec: LayerSpec, **kw) -> LayerSpec:
    """Same workload with some fields replaced (smaller shapes for quick cases)."""
    return dataclasses.replace(spec, **kw)


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (nearest-even) and return the bit patterns."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return u.astype(np.uint16)


def f32_to_f16_bits(a: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float16).view(np.uint16)


def _draw_basis(rng: np.random.Generator, D: int, n: int, method: str = "qr") -> np.ndarray:
    if method == "qr":
        g = rng.standard_normal((D, n)) / math.sqrt(D)
        q, _ = np.linalg.qr(g)          # D x n, orthonormal columns
    else:                               # signed permutation x 2 Householder reflections
        q = np.zeros((D, n), dtype=np.float32)
        q[rng.permutation(D)[:n], np.arange(n)] = rng.choice([-1.0, 1.0], size=n)
        for _ in range(2):
            v = rng.standard_normal(D)
            v = (v / np.linalg.norm(v)).astype(np.float32)
            q -= np.outer(2.0 * v, v @ q)
    return f32_to_bf16_bits(q.astype(np.float32))


_SM_GOLDEN = np.uint64(0x9E3779B97F4A7C15)
_SM_C1 = np.uint64(0xBF58476D1CE4E5B9)
_SM_C2 = np.uint64(0x94D049BB133111EB)


def splitmix64(counter: np.ndarray) -> np.ndarray:
    """SplitMix64 output for each 64-bit counter value (wrapping arithmetic)."""
    with np.errstate(over="ignore"):
        z = counter * _SM_GOLDEN
        z ^= z >> np.uint64(30)
        z *= _SM_C1
        z ^= z >> np.uint64(27)
        z *= _SM_C2
        z ^= z >> np.uint64(31)
    return z


def make_layer(spec: LayerSpec, seed: int = 0, layer_index: int = 0,
               alpha_scale: float = 1.0,
               bits_dist: Optional[Dict[int, float]] = None,
               basis_method: Optional[str] = None) -> Dict[str, np.ndarray]:
    """Draw one packed-format layer as host arrays.

    Returns a dict with
      basis  uint16 [3, D, n]   bf16 bits, basis[h][d, j] = Phi_h[d, j]
      bits   uint8  [3, E, n]
      alpha  float32[3, E, n]
      codes  uint16 [3, E, n, I]  code of element i of unit j (fp16 bits if b == 16)
      scale  uint16 [3, E, n, I // group]  fp16 bits (0 where b in {0, 16})
      zero   uint16 [3, E, n, I // group]  fp16 bits (0 where b in {0, 16})
    plus the integer dims D, E, I, n, group.
    """
    D, E, I, n, group = spec.D, spec.E, spec.I, spec.n, spec.group
    if I % group:
        raise ValueError("I must be a multiple of group")
    ng = I // group
    rng = np.random.default_rng([seed, layer_index, 17])
    method = basis_method or ("householder" if spec.layers > 1 else "qr")
    basis = np.stack([_draw_basis(rng, D, n, method) for _ in range(3)])

    dist = _dist(bits_dist) if bits_dist is not None else spec.bits_dist
    vals = np.array([b for b, _ in dist], dtype=np.uint8)
    probs = np.array([p for _, p in dist], dtype=np.float64)
    probs = probs / probs.sum()
    bits = vals[rng.choice(len(vals), size=(3, E, n), p=probs)]

    # codes: SplitMix64 words of a per-layer counter, cut into 16-bit pieces and
    # masked to b bits; blocks of one (projection, expert) drawn in threads
    codes = np.empty((3, E, n, I), dtype=np.uint16)
    mask = np.where(bits >= 16, 0xFFFF, (1 << bits.astype(np.uint32)) - 1).astype(np.uint16)
    words = (n * I + 3) // 4
    key = int(np.random.SeedSequence([seed, layer_index, 19]).generate_state(1, np.uint64)[0])

    def _draw(q):
        h, e = divmod(q, E)
        ctr = np.arange(words, dtype=np.uint64) + np.uint64((key + q * words) % (1 << 64))
        if int(bits[h, e].max()) <= 4:   # 4-bit fields: 16 codes per word
            ctr = ctr[: (n * I + 15) // 16]
            by = splitmix64(ctr).view(np.uint8)
            nib = np.empty(2 * by.size, dtype=np.uint8)
            nib[0::2] = by & 15
            nib[1::2] = by >> 4
            blk = nib[: n * I].reshape(n, I).astype(np.uint16)
        else:                            # 16-bit fields: 4 codes per word
            blk = splitmix64(ctr).view(np.uint16)[: n * I].reshape(n, I)
        codes[h, e] = blk & mask[h, e][:, None]

    with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        list(ex.map(_draw, range(3 * E)))
    sixteen = bits == 16
    if sixteen.any():
        cnt = int(sixteen.sum())
        v = rng.standard_normal((cnt, I)) / math.sqrt(I)
        codes[sixteen] = f32_to_f16_bits(v.astype(np.float32))

    levels = ((1 << np.minimum(bits, 15).astype(np.int64)) - 1).astype(np.float64)
    quant = (bits > 0) & (bits < 16)
    base = np.where(quant, 2.0 * math.sqrt(3.0 / I) / np.maximum(levels, 1.0), 0.0)
    s = base[..., None] * rng.uniform(0.75, 1.25, size=(3, E, n, ng))
    z = np.where(quant, levels / 2.0, 0.0)[..., None] + rng.uniform(-0.5, 0.5, size=(3, E, n, ng))
    s = np.where(quant[..., None], s, 0.0)
    z = np.where(quant[..., None], z, 0.0)

    j = np.arange(1, n + 1, dtype=np.float64)
    alpha = np.broadcast_to((alpha_scale * j ** -0.5).astype(np.float32), (3, E, n)).copy()

    return dict(D=D, E=E, I=I, n=n, group=group,
                basis=basis, bits=bits, alpha=alpha, codes=codes,
                scale=f32_to_f16_bits(s.astype(np.float32)),
                zero=f32_to_f16_bits(z.astype(np.float32)))


def expert_bias(spec: LayerSpec, seed: int = 0) -> np.ndarray:
    if spec.expert_bias_std <= 0:
        return np.zeros(spec.E, dtype=np.float32)
    rng = np.random.default_rng([seed, 29])
    return rng.normal(0.0, spec.expert_bias_std, size=spec.E).astype(np.float32)


def make_inputs(spec: LayerSpec, T: int, seed: int = 0, step: int = 0) -> Tuple[np.ndarray, np.ndarray]:
    """Activations (bf16 bits, T x D) and router logits (fp32, T x E) for one decode step."""
    rng = np.random.default_rng([seed, 31, T, step])
    x = f32_to_bf16_bits(rng.standard_normal((T, spec.D)).astype(np.float32))
    logits = rng.standard_normal((T, spec.E)).astype(np.float32)
    logits = (logits + expert_bias(spec, seed)[None, :]).astype(np.float32)
    return x, logits


def make_router_weight(spec: LayerSpec, seed: int = 0, layer_index: int = 0) -> np.ndarray:
    """Router matrix W_r (E x D, bf16 bits), N(0, 1/D), for the layer stack."""
    rng = np.random.default_rng([seed, layer_index, 37])
    w = rng.standard_normal((spec.E, spec.D)) / math.sqrt(spec.D)
    return f32_to_bf16_bits(w.astype(np.float32))


def make_hidden(spec: LayerSpec, T: int, seed: int = 0, step: int = 0) -> np.ndarray:
    """Hidden state entering the layer stack (fp32 values of bf16 N(0,1) draws)."""
    rng = np.random.default_rng([seed, 41, T, step])
    xb = f32_to_bf16_bits(rng.standard_normal((T, spec.D)).astype(np.float32))
    return (xb.astype(np.uint32) << 16).view(np.float32)


def permute_units(layer: Dict[str, np.ndarray], perm: Sequence[int]) -> Dict[str, np.ndarray]:
    """Apply one permutation of the unit index j to every per-unit array and to the
    basis columns together (a relabelling of the spectral components)."""
    perm = np.asarray(perm)
    out = dict(layer)
    out["basis"] = np.ascontiguousarray(layer["basis"][:, :, perm])
    for k in ("bits", "alpha", "codes", "scale", "zero"):
        out[k] = np.ascontiguousarray(layer[k][:, :, perm])
    return out


def make_float_units(U: int, I: int, seed: int = 0, bits_dist: Optional[Dict[int, float]] = None,
                     zero_groups: int = 0, group: int = 128) -> Tuple[np.ndarray, np.ndarray]:
    """Unquantised spectral units for the quantiser: U unit-norm Gaussian directions of
    length I (fp32, one per row, like the normalised spectral vectors of the method)
    and a bit-width per unit drawn i.i.d. from `bits_dist` (default: mean 2.0 bits).
    `zero_groups` groups of `group` elements are set to zero (edge cases)."""
    rng = np.random.default_rng([seed, 43, U, I])
    p = rng.standard_normal((U, I))
    p /= np.maximum(np.linalg.norm(p, axis=1, keepdims=True), 1e-300)
    p = p.astype(np.float32)
    if zero_groups and U and I >= group:
        ng = I // group
        for _ in range(zero_groups):
            u, g = int(rng.integers(U)), int(rng.integers(ng))
            p[u, g * group:(g + 1) * group] = 0.0
    dist = _dist(bits_dist if bits_dist is not None else DIST_MEAN_2_0)
    vals = np.array([b for b, _ in dist], dtype=np.uint8)
    probs = np.array([q for _, q in dist], dtype=np.float64)
    bits = vals[rng.choice(len(vals), size=U, p=probs / probs.sum())]
    return p, bits
