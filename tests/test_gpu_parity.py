"""GPU parity of the CUDA forward (through the C ABI) against the fp64 oracle.

Bar: max|y_gpu - y_ref| / ||y_ref||_inf <= 2e-3 (bf16 activations, fp32
accumulation), on the seeded synthetic workloads and on small layers that hit
every bit-width, group size, ragged unit count, padded row block and token
batching path, plus the degenerate cases of the method.
"""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu
TOL = 2e-3


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


def rel_err(y, ref):
    return float(np.max(np.abs(y - ref)) / max(np.max(np.abs(ref)), 1e-30))


def gpu_forward(env, L, x, logits, k):
    torch, bm = env
    xd = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda()
    ld = torch.from_numpy(np.ascontiguousarray(logits)).cuda()
    y = bm.moe_forward(L, xd, ld, k)
    torch.cuda.synchronize()
    return y.cpu().numpy().astype(np.float64)


def check(env, layer, x, logits, k, tol=TOL, L=None):
    torch, bm = env
    own = L is None
    if own:
        L = bm.bitsmoe_pack(layer, device=0)
    y = gpu_forward(env, L, x, logits, k)
    ref = oracle.moe_forward_factored(layer, x, logits, k)
    err = rel_err(y, ref)
    assert err <= tol, err
    if own:
        L.free()
    return err, y, ref


ALL_BITS = {0: 0.1, 1: 0.15, 2: 0.2, 3: 0.15, 4: 0.1, 6: 0.1, 8: 0.1, 16: 0.1}


def small(**kw):
    base = dict(D=96, E=4, I=256, n=72, group=64, top_k=2)
    base.update(kw)
    return synth.scaled_spec(synth.WORKLOADS["tiny"], **base)


# --------------------------------------------------------------------------
def test_tiny_workload(env):
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=0)
    x, logits = synth.make_inputs(spec, 4, seed=0)
    err, y, ref = check(env, layer, x, logits, spec.top_k)
    # the definition (dense reconstruction) agrees too
    dense = oracle.moe_forward_dense(layer, x, logits, spec.top_k)
    assert rel_err(y, dense) <= TOL


def test_tiny_large_amplitude(env):
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=0, alpha_scale=30.0)   # SiLU in its nonlinear range
    x, logits = synth.make_inputs(spec, 4, seed=0)
    check(env, layer, x, logits, spec.top_k)


@pytest.mark.parametrize("group,I", [(32, 96), (64, 256), (128, 384), (256, 512)])
@pytest.mark.parametrize("T", [1, 3, 9])
def test_all_bit_widths_groups_and_token_batches(env, group, I, T):
    spec = small(group=group, I=I, n=75, D=100)        # ragged n and D
    layer = synth.make_layer(spec, seed=group + T, bits_dist=ALL_BITS, alpha_scale=4.0)
    x, logits = synth.make_inputs(spec, T, seed=T)
    check(env, layer, x, logits, spec.top_k)


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8, 16])
def test_uniform_bit_width(env, b):
    """Five tokens: the decode chain with the tensor-core projections."""
    torch, bm = env
    spec = small(n=70)
    layer = synth.make_layer(spec, seed=b, bits_dist={b: 1.0}, alpha_scale=3.0)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_forward_plan(L, 5, spec.top_k) == bm.PLAN_DECODE_CHAIN | bm.PLAN_TC_PROJECTIONS
    assert bm.bitsmoe_forward_plan(L, 3, spec.top_k) & bm.PLAN_FUSED   # one fused forward per token
    x, logits = synth.make_inputs(spec, 5, seed=b)
    check(env, layer, x, logits, spec.top_k, L=L)


def set_unit(layer, h, e, j, b, rng):
    """Give unit (h, e, j) bit-width b with valid codes, scale and zero."""
    layer["bits"][h, e, j] = b
    ng = layer["scale"].shape[-1]
    layer["codes"][h, e, j] = rng.integers(0, 1 << b, layer["I"])
    layer["scale"][h, e, j] = synth.f32_to_f16_bits(np.full(ng, 0.05, np.float32))
    layer["zero"][h, e, j] = synth.f32_to_f16_bits(np.full(ng, ((1 << b) - 1) / 2, np.float32))


def test_evicted_units_and_experts(env):
    spec = small()
    layer = synth.make_layer(spec, seed=5, bits_dist=ALL_BITS, alpha_scale=3.0)
    layer["bits"][:, 1, :] = 0            # expert 1 fully evicted: contributes exactly 0
    layer["bits"][0, 2, :] = 0            # gate of expert 2 evicted: gate = 0 -> h = 0
    layer["bits"][2, 3, :] = 0
    set_unit(layer, 2, 3, 11, 2, np.random.default_rng(0))   # down of expert 3: a single live unit
    x, logits = synth.make_inputs(spec, 6, seed=5)
    logits[:, 1] += 5.0                   # route every token through the evicted expert
    check(env, layer, x, logits, spec.top_k)


def test_unit_permutation_invariance(env):
    torch, bm = env
    spec = small()
    layer = synth.make_layer(spec, seed=8, bits_dist=ALL_BITS, alpha_scale=3.0)
    x, logits = synth.make_inputs(spec, 4, seed=8)
    _, y0, ref = check(env, layer, x, logits, spec.top_k)
    perm = np.random.default_rng(3).permutation(spec.n)
    _, y1, _ = check(env, synth.permute_units(layer, perm), x, logits, spec.top_k)
    assert rel_err(y1, ref) <= TOL
    assert rel_err(y1, y0) <= TOL


def test_routing_ties_and_extreme_k(env):
    spec = small(E=6)
    layer = synth.make_layer(spec, seed=9, alpha_scale=3.0)
    x, _ = synth.make_inputs(spec, 7, seed=9)
    rng = np.random.default_rng(9)
    logits = rng.integers(-2, 3, size=(7, spec.E)).astype(np.float32)   # many exact ties
    for k in (1, 3, spec.E):
        check(env, layer, x, logits, k)


def test_host_buffer_entry_point_matches(env):
    torch, bm = env
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=1)
    x, logits = synth.make_inputs(spec, 4, seed=1)
    L = bm.bitsmoe_pack(layer, device=0)
    ws = bm.Workspace(L, 4, spec.top_k)
    y_host = bm.bitsmoe_moe_forward_host(x, logits, spec.top_k, L, ws.ptr, ws.nbytes,
                                         torch.cuda.current_stream().cuda_stream)
    y_dev = gpu_forward(env, L, x, logits, spec.top_k)
    ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    assert rel_err(y_host.astype(np.float64), ref) <= TOL
    assert rel_err(y_host.astype(np.float64), y_dev) <= 1e-5
    assert bm.bitsmoe_last_device_status(ws.ptr, 0) == 0


def test_host_buffer_single_token_pinned_and_pageable(env):
    """One token on the fused kernel through the host-buffer entry point: pinned buffers are
    read and written by the kernel in place, pageable ones are copied; both match."""
    torch, bm = env
    spec = small()
    layer = synth.make_layer(spec, seed=12, alpha_scale=3.0)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_forward_launches(L, 1, spec.top_k) == 1
    ws = bm.Workspace(L, 1, spec.top_k)
    st = torch.cuda.current_stream().cuda_stream
    for step in range(3):
        x, logits = synth.make_inputs(spec, 1, seed=12, step=step)
        ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
        y_page = bm.bitsmoe_moe_forward_host(x, logits, spec.top_k, L, ws.ptr, ws.nbytes, st)
        xp = torch.from_numpy(x.view(np.int16)).pin_memory()
        lp = torch.from_numpy(logits).pin_memory()
        yp = torch.full((1, spec.D), float("nan"), dtype=torch.float32).pin_memory()
        rc = bm._lib().bitsmoe_moe_forward_host(xp.data_ptr(), lp.data_ptr(), 1, spec.top_k, L.handle,
                                                yp.data_ptr(), ws.ptr, ws.nbytes, st)
        assert rc == 0
        y_pin = yp.numpy().astype(np.float64)
        assert rel_err(y_page.astype(np.float64), ref) <= TOL
        assert rel_err(y_pin, ref) <= TOL
        assert rel_err(y_pin, y_page.astype(np.float64)) <= 1e-5
    assert bm.bitsmoe_last_device_status(ws.ptr, 0) == 0


@pytest.mark.parametrize("T", [1, 3])
def test_host_buffer_async_steps_in_flight(env, T):
    """The asynchronous host-buffer entry point: six steps enqueued back to back on one
    stream and workspace, each with its own pinned input and output buffers (for T = 1 the
    fused kernel reads and writes them in place), one synchronisation at the end; every
    step's output matches the oracle."""
    torch, bm = env
    spec = small()
    layer = synth.make_layer(spec, seed=13, alpha_scale=3.0)
    L = bm.bitsmoe_pack(layer, device=0)
    ws = bm.Workspace(L, T, spec.top_k)
    st = torch.cuda.Stream()
    steps = []
    for step in range(6):
        x, logits = synth.make_inputs(spec, T, seed=13, step=step)
        xp = torch.from_numpy(x.view(np.int16).copy()).pin_memory()
        lp = torch.from_numpy(logits.copy()).pin_memory()
        yp = torch.full((T, spec.D), float("nan"), dtype=torch.float32).pin_memory()
        rc = bm._lib().bitsmoe_moe_forward_host_async(xp.data_ptr(), lp.data_ptr(), T, spec.top_k, L.handle,
                                                      yp.data_ptr(), ws.ptr, ws.nbytes, st.cuda_stream)
        assert rc == 0
        steps.append((x, logits, xp, lp, yp))
    st.synchronize()
    for x, logits, _, _, yp in steps:
        ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
        assert rel_err(yp.numpy().astype(np.float64), ref) <= TOL
    assert bm.bitsmoe_last_device_status(ws.ptr, 0) == 0


def test_blob_upload_and_device_unpack_roundtrip(env):
    torch, bm = env
    spec = small()
    layer = synth.make_layer(spec, seed=10, bits_dist=ALL_BITS)
    blob = bm.bitsmoe_pack_to_host(layer)
    L = bm.bitsmoe_load_blob(blob, device=0)
    out = bm.bitsmoe_unpack(L)
    np.testing.assert_array_equal(out["bits"], layer["bits"])
    live = layer["bits"] > 0
    np.testing.assert_array_equal(out["codes"][live], layer["codes"][live])
    np.testing.assert_array_equal(out["basis"], layer["basis"])
    x, logits = synth.make_inputs(spec, 3, seed=10)
    check(env, layer, x, logits, spec.top_k, L=L)


def test_argument_errors(env):
    torch, bm = env
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=2)
    L = bm.bitsmoe_pack(layer, device=0)
    T, k = 4, spec.top_k
    x = torch.zeros((T, spec.D), dtype=torch.int16, device="cuda")
    lg = torch.zeros((T, spec.E), dtype=torch.float32, device="cuda")
    y = torch.zeros((T, spec.D), dtype=torch.float32, device="cuda")
    ws = bm.Workspace(L, T, k)

    def rc(**kw):
        a = dict(x=x.data_ptr(), lg=lg.data_ptr(), T=T, k=k, y=y.data_ptr(), ws=ws.ptr, wsb=ws.nbytes)
        a.update(kw)
        try:
            bm.bitsmoe_moe_forward(a["x"], a["lg"], a["T"], a["k"], L, a["y"], a["ws"], a["wsb"], 0)
            return 0
        except bm.BitsMoEError as e:
            return e.code

    assert rc() == 0
    assert rc(T=0, x=0, lg=0, y=0) == 0                          # empty batch: no-op
    assert rc(k=0) == bm.ERR_CODE["INVALID_ARG"]
    assert rc(k=spec.E + 1) == bm.ERR_CODE["INVALID_ARG"]
    assert rc(wsb=ws.nbytes - 1) == bm.ERR_CODE["WORKSPACE_TOO_SMALL"]
    assert rc(x=x.data_ptr() + 2) == bm.ERR_CODE["ALIGNMENT"]
    assert rc(ws=ws.ptr + 16) == bm.ERR_CODE["ALIGNMENT"]
    assert rc(y=0) == bm.ERR_CODE["INVALID_ARG"]
    assert bm.bitsmoe_workspace_bytes(L, 4, 0) == 0
    torch.cuda.synchronize()


# --------------------------------------------------------------------------
# the paper-shaped workloads
# --------------------------------------------------------------------------
def test_qw3_decode_batch1(env):
    spec = synth.WORKLOADS["qw3"]
    layer = synth.make_layer(spec, seed=0)
    torch, bm = env
    L = bm.bitsmoe_pack(layer, device=0)
    for step in range(3):
        x, logits = synth.make_inputs(spec, 1, seed=0, step=step)
        check(env, layer, x, logits, spec.top_k, L=L)


def test_qw3_skewed_load_batches(env):
    spec = synth.WORKLOADS["qw3_skew"]
    layer = synth.make_layer(spec, seed=0)
    torch, bm = env
    L = bm.bitsmoe_pack(layer, device=0)
    for T in spec.tokens:
        x, logits = synth.make_inputs(spec, T, seed=0)
        if T <= 32:
            check(env, layer, x, logits, spec.top_k, L=L)
        else:
            # full batch on the GPU, oracle on a sample of tokens (tokens are independent)
            y = gpu_forward(env, L, x, logits, spec.top_k)
            rows = np.random.default_rng(T).choice(T, 12, replace=False)
            ref = oracle.moe_forward_factored(layer, x[rows], logits[rows], spec.top_k)
            assert rel_err(y[rows], ref) <= TOL


def test_mixtral_shape(env):
    spec = synth.WORKLOADS["mixtral"]
    layer = synth.make_layer(spec, seed=0)
    torch, bm = env
    L = bm.bitsmoe_pack(layer, device=0)
    for T in spec.tokens:
        x, logits = synth.make_inputs(spec, T, seed=0)
        check(env, layer, x, logits, spec.top_k, L=L)


@pytest.mark.parametrize("T", [1, 2, 3])
def test_decode_chain_without_fused_plan(env, T):
    """A layer whose per-block shares do not fit the fused kernel (D = n = 4096): one to
    three tokens take the decode chain with the bulk-copy GEMV projections."""
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["mixtral"], E=3, I=256, top_k=2)
    layer = synth.make_layer(spec, seed=40 + T)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_forward_plan(L, T, spec.top_k) == bm.PLAN_DECODE_CHAIN
    x, logits = synth.make_inputs(spec, T, seed=40 + T)
    check(env, layer, x, logits, spec.top_k, L=L)
