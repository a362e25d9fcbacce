"""The offline steps compose (no GPU needed): float spectral units -> bit allocation under
the paper's budget -> quantiser -> the library's host packer -> bit-exact unpack, and the
forward on the packed layer approaches the float layer as the budget grows.  The
allocation and the quantiser here are the oracles (the GPU kernels equal them bit for bit,
tests/test_gpu_allocate.py and tests/test_gpu_quantize.py); the packer is the library's."""
import os

import numpy as np
import pytest

import oracle
import synth
from oracle import allocator as A
from oracle import quantizer as Q

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


@pytest.fixture(scope="module")
def bm():
    import __graft_entry__
    __graft_entry__.build_library()
    import paper_2606_00079_gb300 as bm
    return bm


def _kappa():
    out = {}
    with open(os.path.join(GOLDEN, "kappa_values.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                out[int(k)] = float(v)
    return out


def _quantised_layer(spec, P, bits, layer):
    shp = (3, spec.E, spec.n)
    codes, scale, zero = Q.quantize_units(P, bits, spec.group)
    return dict(layer, bits=bits.reshape(shp).astype(np.uint8), codes=codes.reshape(*shp, spec.I),
                scale=scale.reshape(*shp, -1), zero=zero.reshape(*shp, -1))


def test_allocate_quantise_pack_unpack_forward(bm):
    # E n b_eq - 16 n^2 / I must be positive: at 8 x 64 units of 512 the bases cost 128 unit-bits
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=64, E=8, I=512, n=64, group=64, top_k=2)
    layer = synth.make_layer(spec, seed=21)
    U = spec.E * spec.n
    P, _ = synth.make_float_units(3 * U, spec.I, seed=21)
    alpha = layer["alpha"].reshape(-1)
    beta = np.random.default_rng(21).lognormal(0.0, 1.0, 3 * U).astype(np.float32)
    x, logits = synth.make_inputs(spec, 3, seed=21)
    flt = dict(layer, bits=np.full((3, spec.E, spec.n), 16, np.uint8),
               codes=P.astype(np.float16).view(np.uint16).reshape(3, spec.E, spec.n, spec.I))
    y_float = oracle.moe_forward_dense(flt, x, logits, spec.top_k)
    errs = []
    for b_eq in (1.5, 2.5, 4.0, 6.0):
        B = A.projection_budget(spec.E, spec.n, spec.I, b_eq)
        bits = np.concatenate([A.allocate(A.costs(P[h * U:(h + 1) * U], alpha[h * U:(h + 1) * U],
                                                  beta[h * U:(h + 1) * U], 0.5, _kappa()), B)
                               for h in range(3)])
        for h in range(3):
            assert int(bits[h * U:(h + 1) * U].astype(np.int64).sum()) <= B
        q = _quantised_layer(spec, P, bits, layer)
        blob = bm.bitsmoe_pack_to_host(q)                      # the packer accepts the quantiser's output
        back = bm.bitsmoe_unpack_blob(blob, (spec.D, spec.E, spec.I, spec.n, spec.group))
        live = q["bits"] > 0
        np.testing.assert_array_equal(back["bits"], q["bits"])
        np.testing.assert_array_equal(back["codes"][live], q["codes"][live])
        quant = live & (q["bits"] < 16)
        np.testing.assert_array_equal(back["scale"][quant], q["scale"][quant])
        np.testing.assert_array_equal(back["zero"][quant], q["zero"][quant])
        y = oracle.moe_forward_dense(q, x, logits, spec.top_k)
        errs.append(float(np.max(np.abs(y - y_float)) / np.max(np.abs(y_float))))
    assert all(b < a for a, b in zip(errs, errs[1:])), errs    # more bits, closer to the float layer
    assert errs[-1] < 0.1, errs
