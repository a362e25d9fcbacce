"""GPU parity of the per-unit quantiser (bitsmoe_quantize_units, through the C ABI)
against the quantiser oracle (oracle/quantizer.py).

The quantiser turns float spectral units into integer codes, so the bar is
bit-exact: codes, fp16 scales and fp16 zeros must equal the oracle's for every
bit-width, group size and candidate grid, on ragged unit counts, all-zero
groups and a layer-sized sample; a unit with an unsupported bit-width gets
zero outputs and the status word.  A layer quantised on the GPU, packed and run
through the forward matches the forward oracle on the oracle-quantised layer.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle import quantizer as Q

pytestmark = pytest.mark.gpu
TOL = 2e-3
ALL_BITS = {0: .05, 1: .15, 2: .25, 3: .2, 4: .15, 6: .08, 8: .07, 16: .05}


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00079_gb300 as bm
    torch.cuda.set_device(0)
    return torch, bm


def gpu_quantize(env, P, bits, group, grid):
    torch, bm = env
    pd = torch.from_numpy(np.ascontiguousarray(P, dtype=np.float32)).cuda()
    bd = torch.from_numpy(np.ascontiguousarray(bits, dtype=np.uint8)).cuda()
    codes, scale, zero, status = bm.quantize_units(pd, bd, group, grid)
    torch.cuda.synchronize()
    u16 = lambda t: t.cpu().numpy().view(np.uint16)
    return u16(codes), u16(scale), u16(zero), int(status.item())


def assert_same(got, want):
    for name, g, w in zip(("codes", "scale", "zero"), got, want):
        if not np.array_equal(g, w):
            bad = np.argwhere(g != w)
            raise AssertionError(f"{name}: {len(bad)} mismatches, first at {bad[:5].tolist()}: "
                                 f"{g[tuple(bad[0])]} != {w[tuple(bad[0])]}")


@pytest.mark.parametrize("U,I,group,grid,seed", [
    (37, 256, 64, 256, 0),      # ragged unit count, every bit-width
    (129, 768, 128, 256, 1),    # Qwen3-shaped unit length, group 128
    (64, 512, 32, 32, 2),       # smallest group and grid
    (16, 1024, 256, 1024, 3),   # largest group and grid
    (33, 384, 128, 64, 4),
    (5, 128, 128, 512, 5),
])
def test_quantizer_matches_oracle_bit_exactly(env, U, I, group, grid, seed):
    P, bits = synth.make_float_units(U, I, seed=seed, bits_dist=ALL_BITS, zero_groups=3, group=group)
    got = gpu_quantize(env, P, bits, group, grid)
    assert got[3] == 0
    assert_same(got[:3], Q.quantize_units(P, bits, group, grid))


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8, 16, 0])
def test_uniform_bit_width(env, b):
    P, _ = synth.make_float_units(48, 256, seed=10 + b)
    bits = np.full(48, b, np.uint8)
    assert_same(gpu_quantize(env, P, bits, 64, 256)[:3], Q.quantize_units(P, bits, 64, 256))


def test_scaled_and_extreme_values(env):
    """Inputs far from unit norm: tiny (fp16 subnormal scales), large (scales near the fp16
    limit, skipped candidates), exact zeros and negative zeros."""
    P, bits = synth.make_float_units(96, 256, seed=7, bits_dist=ALL_BITS)
    P[:32] *= np.float32(2.0 ** -18)
    P[32:64] *= np.float32(3.0e4)
    P[64, :64] = 0.0
    P[65, :64] = -0.0
    assert_same(gpu_quantize(env, P, bits, 64, 128)[:3], Q.quantize_units(P, bits, 64, 128))


def test_layer_sized_sample(env):
    """One Qwen3-shaped expert's worth of units (3 x 2048 units of 768, group 128, mean 2.0
    bits) in one launch; every 12th unit compared with the oracle."""
    U, I = 3 * 2048, 768
    P, bits = synth.make_float_units(U, I, seed=11)
    codes, scale, zero, status = gpu_quantize(env, P, bits, 128, 256)
    assert status == 0
    idx = np.arange(0, U, 12)
    assert_same((codes[idx], scale[idx], zero[idx]), Q.quantize_units(P[idx], bits[idx], 128, 256))


def test_unsupported_bits_zero_outputs_and_status(env):
    torch, bm = env
    P, _ = synth.make_float_units(8, 128, seed=12)
    bits = np.array([2, 5, 3, 7, 2, 9, 4, 255], np.uint8)
    codes, scale, zero, status = gpu_quantize(env, P, bits, 64, 64)
    assert status == bm.ERR_CODE["UNSUPPORTED_BITS"]
    bad = np.array([1, 3, 5, 7])
    assert not codes[bad].any() and not scale[bad].any() and not zero[bad].any()
    good = np.array([0, 2, 4, 6])
    assert_same((codes[good], scale[good], zero[good]), Q.quantize_units(P[good], bits[good], 64, 64))


def test_empty_call_is_a_no_op(env):
    torch, bm = env
    bm.bitsmoe_quantize_units(0, 0, 0, 128, 64, 256, 0, 0, 0, 0, 0)


def test_gpu_quantised_layer_runs_through_the_forward(env):
    """Float units -> GPU quantiser -> bitsmoe_pack -> forward, against the forward oracle
    on the oracle-quantised layer (the same stored layer, so the forward's own bar)."""
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=256, E=8, I=512, n=256, group=64, top_k=2)
    layer = synth.make_layer(spec, seed=13)
    U = 3 * spec.E * spec.n
    P, bits = synth.make_float_units(U, spec.I, seed=13, group=spec.group, zero_groups=4)
    codes, scale, zero, status = gpu_quantize(env, P, bits, spec.group, 256)
    assert status == 0
    shp = (3, spec.E, spec.n)
    q = dict(layer, bits=bits.reshape(shp), codes=codes.reshape(*shp, spec.I),
             scale=scale.reshape(*shp, -1), zero=zero.reshape(*shp, -1))
    oc, osc, oz = Q.quantize_units(P, bits, spec.group, 256)
    qo = dict(layer, bits=bits.reshape(shp), codes=oc.reshape(*shp, spec.I),
              scale=osc.reshape(*shp, -1), zero=oz.reshape(*shp, -1))
    L = bm.bitsmoe_pack(q, device=0)
    x, logits = synth.make_inputs(spec, 4, seed=13)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ld = torch.from_numpy(logits).cuda()
    y = bm.moe_forward(L, xd, ld, spec.top_k)
    torch.cuda.synchronize()
    ref = oracle.moe_forward_dense(qo, x, logits, spec.top_k)
    err = float(np.max(np.abs(y.cpu().numpy() - ref)) / np.max(np.abs(ref)))
    assert err <= TOL, err
