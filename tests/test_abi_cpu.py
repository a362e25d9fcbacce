"""Host-side checks of the C-ABI library (no GPU needed).

* the library loads and exports every function include/bitsmoe.h declares;
* packing into the bucketed layout and unpacking it round-trips bit-exactly,
  for every bit-width, group size, ragged unit counts, padded rows and the
  degenerate layers (an expert with every unit evicted, a single live unit);
* malformed inputs and blobs are rejected with the documented error codes.
"""
import os
import re

import numpy as np
import pytest

import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bm():
    import __graft_entry__
    __graft_entry__.build_library()
    import paper_2606_00079_gb300 as bm
    return bm


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "bitsmoe.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(bitsmoe_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(bm):
    lib = bm._lib()
    declared = _declared_functions()
    assert len(declared) >= 15
    for name in declared:
        assert hasattr(lib, name), name
    assert set(declared) == set(bm.SIGNATURES), "binding signatures differ from the header"


def _spec(**kw):
    base = dict(D=48, E=3, I=256, n=40, group=64, top_k=2)
    base.update(kw)
    return synth.scaled_spec(synth.WORKLOADS["tiny"], **base)


def _expect_roundtrip(layer, out):
    """Compare what is stored: every bit-width, basis, alpha of live units, codes of
    live units, scale/zero of quantised units (evicted units unpack as zeros)."""
    np.testing.assert_array_equal(out["basis"], layer["basis"])
    np.testing.assert_array_equal(out["bits"], layer["bits"])
    live = layer["bits"] > 0
    np.testing.assert_array_equal(out["alpha"][live], layer["alpha"][live])
    assert not out["alpha"][~live].any()
    np.testing.assert_array_equal(out["codes"][live], layer["codes"][live])
    assert not out["codes"][~live].any()
    quant = live & (layer["bits"] < 16)
    np.testing.assert_array_equal(out["scale"][quant], layer["scale"][quant])
    np.testing.assert_array_equal(out["zero"][quant], layer["zero"][quant])
    assert not out["scale"][~quant].any()


ALL_BITS = {0: 0.1, 1: 0.15, 2: 0.2, 3: 0.15, 4: 0.1, 6: 0.1, 8: 0.1, 16: 0.1}


@pytest.mark.parametrize("group,I", [(32, 96), (64, 256), (128, 384), (256, 512)])
def test_pack_roundtrip_all_bit_widths(bm, group, I):
    spec = _spec(group=group, I=I)
    layer = synth.make_layer(spec, seed=group, bits_dist=ALL_BITS)
    blob = bm.bitsmoe_pack_to_host(layer)
    out = bm.bitsmoe_unpack_blob(blob, (spec.D, spec.E, spec.I, spec.n, spec.group))
    _expect_roundtrip(layer, out)


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8, 16])
def test_pack_roundtrip_uniform_and_ragged(bm, b):
    # n = 37 units: ragged against every tile width (2, 4, 8, 16, 32)
    spec = _spec(n=37, D=40)
    layer = synth.make_layer(spec, seed=b, bits_dist={b: 1.0})
    out = bm.bitsmoe_unpack_blob(bm.bitsmoe_pack_to_host(layer), (spec.D, spec.E, spec.I, spec.n, spec.group))
    _expect_roundtrip(layer, out)


def test_pack_roundtrip_degenerate_layers(bm):
    spec = _spec()
    layer = synth.make_layer(spec, seed=1, bits_dist=ALL_BITS)
    layer["bits"][0, 1, :] = 0            # gate of expert 1: every unit evicted
    layer["bits"][2, 0, :] = 0            # down of expert 0: a single live unit
    layer["bits"][2, 0, 17] = 3
    layer["codes"][2, 0, 17] = np.arange(spec.I) % 8
    layer["scale"][2, 0, 17] = 0x2C00
    layer["zero"][2, 0, 17] = 0x4300
    layer["bits"][:, 2, :] = 0            # expert 2 entirely evicted
    out = bm.bitsmoe_unpack_blob(bm.bitsmoe_pack_to_host(layer), (spec.D, spec.E, spec.I, spec.n, spec.group))
    _expect_roundtrip(layer, out)


def test_pack_roundtrip_tiny_workload(bm):
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=0)
    blob = bm.bitsmoe_pack_to_host(layer)
    out = bm.bitsmoe_unpack_blob(blob, (spec.D, spec.E, spec.I, spec.n, spec.group))
    _expect_roundtrip(layer, out)
    # packing is deterministic
    np.testing.assert_array_equal(bm.bitsmoe_pack_to_host(layer), blob)


def test_invalid_inputs_rejected(bm):
    spec = _spec()
    layer = synth.make_layer(spec, seed=2)
    bad = dict(layer)
    bad["bits"] = layer["bits"].copy()
    bad["bits"][1, 0, 3] = 5
    with pytest.raises(bm.BitsMoEError) as ei:
        bm.bitsmoe_pack_to_host(bad)
    assert ei.value.code == bm.ERR_CODE["UNSUPPORTED_BITS"]
    bad = dict(layer)
    bad["codes"] = layer["codes"].copy()
    j = int(np.argmax(layer["bits"][0, 0] == 2))
    assert layer["bits"][0, 0, j] == 2
    bad["codes"][0, 0, j, 5] = 4               # code out of range for a 2-bit unit
    with pytest.raises(bm.BitsMoEError) as ei:
        bm.bitsmoe_pack_to_host(bad)
    assert ei.value.code == bm.ERR_CODE["INVALID_ARG"]
    bad = dict(layer, group=48)
    with pytest.raises(bm.BitsMoEError) as ei:
        bm.bitsmoe_pack_to_host(bad)
    assert ei.value.code == bm.ERR_CODE["SHAPE"]
    bad = dict(layer, I=250)                 # not a multiple of the group
    with pytest.raises(bm.BitsMoEError) as ei:
        bm.bitsmoe_pack_to_host(bad)
    assert ei.value.code == bm.ERR_CODE["SHAPE"]


def test_malformed_blob_rejected(bm):
    spec = _spec()
    layer = synth.make_layer(spec, seed=3)
    blob = bm.bitsmoe_pack_to_host(layer)
    dims = (spec.D, spec.E, spec.I, spec.n, spec.group)
    for mutate in ("magic", "truncate", "offset", "unit"):
        b = blob.copy()
        if mutate == "magic":
            b[0] ^= 0xFF
        elif mutate == "truncate":
            b = b[:-256]
        elif mutate == "offset":
            # ImageHeader: 2 u32 + 14 i32 = 64 bytes, then total_bytes, off_desc, ...
            off = np.frombuffer(b[72:80].tobytes(), np.uint64)[0]
            b[72:80] = np.frombuffer(np.uint64(off + 10 ** 9).tobytes(), np.uint8)
        else:
            # first unit index of the first (h, e) block: set it out of range
            desc_off = int(np.frombuffer(b[72:80].tobytes(), np.uint64)[0])
            unit_off = int(np.frombuffer(b[desc_off + 48:desc_off + 56].tobytes(), np.uint64)[0])
            b[unit_off:unit_off + 4] = np.frombuffer(np.int32(10 ** 6).tobytes(), np.uint8)
        with pytest.raises(bm.BitsMoEError) as ei:
            bm.bitsmoe_unpack_blob(b, dims)
        assert ei.value.code == bm.ERR_CODE["BLOB"], mutate


def test_strerror(bm):
    assert bm.bitsmoe_strerror(0) == "ok"
    assert "workspace" in bm.bitsmoe_strerror(-4)


def test_quantize_units_host_checks(bm):
    """bitsmoe_quantize_units rejects bad arguments on the host, before any device work."""
    lib = bm._lib()
    A = 4096   # a 16-byte-aligned stand-in address (never dereferenced: the checks fail first)
    q = lambda U, I, group, grid, p=A, codes=A, scale=A: lib.bitsmoe_quantize_units(
        p, A, U, I, group, grid, codes, scale, A, 0, 0)
    assert q(0, 128, 64, 256) == 0                                   # U == 0: no-op
    assert q(-1, 128, 64, 256) == bm.ERR_CODE["INVALID_ARG"]
    assert q(4, 0, 64, 256) == bm.ERR_CODE["INVALID_ARG"]
    assert q(4, 96, 64, 256) == bm.ERR_CODE["SHAPE"]                 # I % group
    assert q(4, 96, 48, 256) == bm.ERR_CODE["SHAPE"]                 # unsupported group
    assert q(4, 128, 64, 100) == bm.ERR_CODE["INVALID_ARG"]          # grid not in the set
    assert q(4, 128, 64, 2048) == bm.ERR_CODE["INVALID_ARG"]
    assert q(4, 128, 64, 256, p=0) == bm.ERR_CODE["INVALID_ARG"]
    assert q(4, 128, 64, 256, p=A + 4) == bm.ERR_CODE["ALIGNMENT"]
    assert q(4, 128, 64, 256, codes=A + 8) == bm.ERR_CODE["ALIGNMENT"]
    assert q(4, 128, 64, 256, scale=A + 1) == bm.ERR_CODE["ALIGNMENT"]


def test_allocate_bits_host_checks(bm):
    """bitsmoe_allocate_bits rejects bad arguments on the host, before any device work."""
    import ctypes
    lib = bm._lib()
    A = 4096
    k = (ctypes.c_float * 3)(0.149492, 0.0406789, 0.01184786)
    nb = bm.bitsmoe_allocate_workspace_bytes(100)
    assert nb > 100 * 64 and bm.bitsmoe_allocate_workspace_bytes(-1) == 0
    call = lambda U=100, d=64, gamma=0.5, budget=50, p=A, ws=A, wsb=nb, kap=k: lib.bitsmoe_allocate_bits(
        p, A, A, gamma, U, d, kap, budget, A, ws, wsb, 0)
    assert call(U=0) == 0                                            # no-op
    assert call(U=-1) == bm.ERR_CODE["INVALID_ARG"]
    assert call(d=0) == bm.ERR_CODE["INVALID_ARG"]
    assert call(budget=-1) == bm.ERR_CODE["INVALID_ARG"]
    assert call(gamma=1.5) == bm.ERR_CODE["INVALID_ARG"]
    assert call(gamma=float("nan")) == bm.ERR_CODE["INVALID_ARG"]
    assert call(U=1 << 32) == bm.ERR_CODE["SHAPE"]
    assert call(p=0) == bm.ERR_CODE["INVALID_ARG"]
    assert call(kap=None) == bm.ERR_CODE["INVALID_ARG"]
    assert call(p=A + 4) == bm.ERR_CODE["ALIGNMENT"]
    assert call(ws=A + 16) == bm.ERR_CODE["ALIGNMENT"]
    assert call(wsb=nb - 1) == bm.ERR_CODE["WORKSPACE_TOO_SMALL"]


def test_projection_budget_matches_the_formula(bm):
    """bitsmoe_projection_budget (host only) against hand values and the oracle's exact
    rational evaluation of Eq. app_projection_normalized_budget."""
    from oracle import allocator as A
    assert bm.bitsmoe_projection_budget(128, 2048, 768, 2.0) == 436906
    assert bm.bitsmoe_projection_budget(8, 4096, 14336, 2.0) == 46811
    assert bm.bitsmoe_projection_budget(4, 64, 128, 1.5) == -128           # bases exceed the target
    assert bm.bitsmoe_projection_budget(3, 7, 5, (7, 3)) == -108           # floor(49 - 784/5) = floor(-107.8)
    rng = np.random.default_rng(0)
    for _ in range(300):
        E, n, m = int(rng.integers(1, 300)), int(rng.integers(1, 5000)), int(rng.integers(1, 20000))
        beq = round(float(rng.uniform(0, 8)), 3)
        assert bm.bitsmoe_projection_budget(E, n, m, beq) == A.projection_budget(E, n, m, beq), (E, n, m, beq)
    lib = bm._lib()
    import ctypes
    out = ctypes.c_int64()
    assert lib.bitsmoe_projection_budget(0, 1, 1, 1, 1, ctypes.byref(out)) == bm.ERR_CODE["INVALID_ARG"]
    assert lib.bitsmoe_projection_budget(1, 1, 1, 1, 0, ctypes.byref(out)) == bm.ERR_CODE["INVALID_ARG"]
    assert lib.bitsmoe_projection_budget(1, 1, 1, -1, 1, ctypes.byref(out)) == bm.ERR_CODE["INVALID_ARG"]
    assert lib.bitsmoe_projection_budget(1, 1, 1, 1, 1, None) == bm.ERR_CODE["INVALID_ARG"]
    assert lib.bitsmoe_projection_budget(1 << 21, 1, 1, 1, 1, ctypes.byref(out)) == bm.ERR_CODE["SHAPE"]

