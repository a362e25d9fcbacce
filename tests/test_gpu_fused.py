"""GPU parity of the fused single-token decode kernel (one persistent kernel
with grid barriers) against the fp64 oracle.

The fused path runs whenever T == 1 and the layer's per-block shares fit in
shared memory; these cases check that it was taken and cover every bit-width,
group size, evicted units and experts, extreme top-k, consecutive calls and
different layers on one workspace, a workspace that was not zero-filled (the
call must refuse it with a status, not compute), and replay from a CUDA graph.
Bar: max|y_gpu - y_ref| / ||y_ref||_inf <= 2e-3.
"""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu
TOL = 2e-3
ALL_BITS = {0: 0.1, 1: 0.15, 2: 0.2, 3: 0.15, 4: 0.1, 6: 0.1, 8: 0.1, 16: 0.1}


@pytest.fixture(scope="module", params=["clustered", "plain"])
def env(request):
    """Every case runs on both single-token kernels, each forced through the testing hook: the
    clustered one and the one without clusters."""
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    import paper_2606_00079_gb300 as bm
    torch.cuda.set_device(0)
    bm.bitsmoe_debug_single_token_kernel(1 if request.param == "plain" else 2)
    yield torch, bm, request.param
    bm.bitsmoe_debug_single_token_kernel(0)


def rel_err(y, ref):
    return float(np.max(np.abs(y - ref)) / max(np.max(np.abs(ref)), 1e-30))


def small(**kw):
    base = dict(D=96, E=4, I=256, n=72, group=64, top_k=2)
    base.update(kw)
    return synth.scaled_spec(synth.WORKLOADS["tiny"], **base)


def run(env, L, x, logits, k, ws=None):
    torch, bm, kern = env
    assert bm.bitsmoe_forward_launches(L, x.shape[0], k) == 1, "fused path not taken"
    plan = bm.bitsmoe_forward_plan(L, x.shape[0], k)
    assert plan == bm.PLAN_FUSED | (bm.PLAN_CLUSTERED if kern == "clustered" else 0), plan
    xd = torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).cuda()
    ld = torch.from_numpy(np.ascontiguousarray(logits)).cuda()
    if ws is None:
        ws = bm.Workspace(L, x.shape[0], k)
    y = bm.moe_forward(L, xd, ld, k, ws=ws)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    return y.cpu().numpy().astype(np.float64)


def plain_forward(bm, L, x, lg, k, ws, kern):
    """The forward on the fused kernel without clusters (the one pre-norm blocks use), so that
    a block's update can be compared with it up to the order of float atomics."""
    bm.bitsmoe_debug_single_token_kernel(1)
    try:
        return bm.moe_forward(L, x, lg, k, ws=ws)
    finally:
        bm.bitsmoe_debug_single_token_kernel(1 if kern == "plain" else 2)


def check(env, layer, x, logits, k, L=None, ws=None):
    torch, bm, _ = env
    L = L or bm.bitsmoe_pack(layer, device=0)
    y = run(env, L, x, logits, k, ws)
    ref = oracle.moe_forward_factored(layer, x, logits, k)
    err = rel_err(y, ref)
    assert err <= TOL, err
    return y, ref


@pytest.mark.parametrize("b", [1, 2, 3, 4, 6, 8, 16])
def test_fused_uniform_bit_width(env, b):
    spec = small(n=70)
    layer = synth.make_layer(spec, seed=b, bits_dist={b: 1.0}, alpha_scale=3.0)
    x, logits = synth.make_inputs(spec, 1, seed=b)
    check(env, layer, x, logits, spec.top_k)


@pytest.mark.parametrize("group,I", [(32, 96), (64, 256), (128, 384), (256, 512)])
def test_fused_all_bit_widths_and_groups(env, group, I):
    spec = small(group=group, I=I, n=75, D=100, E=8, top_k=3)
    layer = synth.make_layer(spec, seed=group, bits_dist=ALL_BITS, alpha_scale=4.0)
    x, logits = synth.make_inputs(spec, 1, seed=group)
    check(env, layer, x, logits, spec.top_k)


def test_fused_evicted_units_and_experts(env):
    spec = small()
    layer = synth.make_layer(spec, seed=5, bits_dist=ALL_BITS, alpha_scale=3.0)
    layer["bits"][:, 1, :] = 0            # expert 1 fully evicted
    layer["bits"][0, 2, :] = 0            # gate of expert 2 evicted: h = 0
    x, logits = synth.make_inputs(spec, 1, seed=5)
    for route in ((1, 2), (1, 3), (2, 0)):
        lg = logits.copy()
        lg[0, list(route)] += 10.0
        check(env, layer, x, lg, spec.top_k)


def test_fused_top1_and_all_experts(env):
    spec = small(E=6)
    layer = synth.make_layer(spec, seed=9, bits_dist=ALL_BITS, alpha_scale=3.0)
    x, _ = synth.make_inputs(spec, 1, seed=9)
    logits = np.array([[1.0, 2.0, 2.0, -1.0, 2.0, 0.0]], np.float32)   # ties
    torch, bm, kern = env
    L = bm.bitsmoe_pack(layer, device=0)
    for k in (1, 2, spec.E):
        check(env, layer, x, logits, k, L=L)


@pytest.mark.parametrize("E", [33, 200, 256])
def test_fused_routing_ties_many_experts(env, E):
    """Routing inside the fused kernel with several keys per lane (E > 32), ragged
    E, many exact ties and signed zeros: the k largest logits, ties to the lower index."""
    spec = small(E=E, n=40, I=128)
    layer = synth.make_layer(spec, seed=E)
    x, _ = synth.make_inputs(spec, 1, seed=E)
    rng = np.random.default_rng(E)
    logits = rng.integers(-2, 3, size=(1, E)).astype(np.float32)
    logits[0, rng.integers(0, E, size=4)] = -0.0
    torch, bm, kern = env
    L = bm.bitsmoe_pack(layer, device=0)
    for k in (1, 8, 32):
        check(env, layer, x, logits, k, L=L)


def test_fused_consecutive_calls_layers_and_workspace_state(env):
    torch, bm, kern = env
    spec = synth.scaled_spec(synth.WORKLOADS["qw3"], D=512, E=32, I=384, n=512, top_k=4)
    layers = [synth.make_layer(spec, seed=s) for s in (21, 22)]
    Ls = [bm.bitsmoe_pack(l, device=0) for l in layers]
    ws = bm.Workspace(Ls[0], 1, spec.top_k)
    # a workspace that was not zero-filled: the call reports it and leaves y alone
    ws.buf.fill_(0xA5)
    x, logits = synth.make_inputs(spec, 1, seed=3, step=0)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ld = torch.from_numpy(logits).cuda()
    y = torch.full((1, spec.D), 7.0, dtype=torch.float32, device="cuda")
    bm.moe_forward(Ls[0], xd, ld, spec.top_k, ws=ws, y=y)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == bm.ERR_CODE["WORKSPACE_STATE"]
    assert bool((y == 7.0).all())
    # zero-filled: consecutive calls on two layers share it (each call leaves the next one's counters clear)
    ws.buf.zero_()
    for step in range(6):
        i = step % 2
        x, logits = synth.make_inputs(spec, 1, seed=3, step=step)
        check(env, layers[i], x, logits, spec.top_k, L=Ls[i], ws=ws)
    # a multi-token call (kernel chain) on the same workspace does not disturb the counters
    ws4 = bm.Workspace(Ls[0], 4, spec.top_k)
    x4, l4 = synth.make_inputs(spec, 4, seed=3, step=9)
    y4 = bm.moe_forward(Ls[0], torch.from_numpy(x4.view(np.int16)).cuda(), torch.from_numpy(l4).cuda(),
                        spec.top_k, ws=ws4)
    x, logits = synth.make_inputs(spec, 1, seed=3, step=10)
    check(env, layers[0], x, logits, spec.top_k, L=Ls[0], ws=ws4)
    ref4 = oracle.moe_forward_factored(layers[0], x4, l4, spec.top_k)
    assert rel_err(y4.cpu().numpy().astype(np.float64), ref4) <= TOL


def test_fused_graph_replay(env):
    torch, bm, kern = env
    spec = synth.scaled_spec(synth.WORKLOADS["qw3"], D=512, E=32, I=384, n=512, top_k=4)
    layer = synth.make_layer(spec, seed=31)
    L = bm.bitsmoe_pack(layer, device=0)
    ws = bm.Workspace(L, 1, spec.top_k)
    xd = torch.zeros((1, spec.D), dtype=torch.int16, device="cuda")
    ld = torch.zeros((1, spec.E), dtype=torch.float32, device="cuda")
    ys = [torch.zeros((1, spec.D), dtype=torch.float32, device="cuda") for _ in range(3)]
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):        # warm-up outside the capture
        bm.moe_forward(L, xd, ld, spec.top_k, ws=ws, y=ys[0], stream=stream)
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        for y in ys:                       # three forwards back to back in one graph
            bm.moe_forward(L, xd, ld, spec.top_k, ws=ws, y=y, stream=stream)
    for step in range(3):
        x, logits = synth.make_inputs(spec, 1, seed=4, step=step)
        xd.copy_(torch.from_numpy(x.view(np.int16)))
        ld.copy_(torch.from_numpy(logits))
        g.replay()
        torch.cuda.synchronize()
        ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
        for y in ys:
            assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0


def test_fused_plan_taken_for_qw3_dims_not_for_d4096(env):
    torch, bm, kern = env
    qw3 = synth.scaled_spec(synth.WORKLOADS["qw3"], E=8, top_k=8)   # full qw3 dims, fewer experts
    L = bm.bitsmoe_pack(synth.make_layer(qw3, seed=1), device=0)
    assert bm.bitsmoe_forward_launches(L, 1, 8) == 1
    assert bm.bitsmoe_forward_launches(L, 2, 8) == 2   # one fused forward per token
    assert bm.bitsmoe_forward_launches(L, 5, 8) == 5
    # D = n = 4096: a block's share of the input bases (54 rows of 8 KB) exceeds shared memory
    big = synth.scaled_spec(synth.WORKLOADS["mixtral"], E=2, I=128, top_k=1)
    Lb = bm.bitsmoe_pack(synth.make_layer(big, seed=1), device=0)
    assert bm.bitsmoe_forward_launches(Lb, 1, 1) == 5


@pytest.mark.parametrize("E,top_k", [(4, 2), (200, 8)])
def test_block_forward_fused_norm(env, E, top_k):
    """A one-token pre-norm block runs as the single fused kernel, which also
    computes the RMSNorm and the router logits (E = 200 > blocks: two router
    rows on some blocks).  Its update must match the two-step path
    (norm/router kernel, then the forward) up to the order of the float
    atomics, and the oracle's MoE on the same x and logits."""
    torch, bm, kern = env
    spec = small(E=E, top_k=top_k, n=72)
    layer = synth.make_layer(spec, seed=5)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_block_forward_launches(L, 1, top_k) == 1
    assert bm.bitsmoe_block_forward_launches(L, 2, top_k) == 2
    assert bm.bitsmoe_block_forward_launches(L, 5, top_k) == bm.bitsmoe_forward_launches(L, 5, top_k) + 1
    wr = torch.from_numpy(synth.make_router_weight(spec, seed=5).view(np.int16)).cuda()
    h0 = torch.from_numpy(synth.make_hidden(spec, 1, seed=5)).cuda() * 3.0
    eps, st = 1e-6, torch.cuda.current_stream().cuda_stream
    ws = bm.Workspace(L, 1, top_k)
    x = torch.empty((1, spec.D), dtype=torch.int16, device="cuda")
    lg = torch.empty((1, spec.E), dtype=torch.float32, device="cuda")
    bm.bitsmoe_rmsnorm_router(h0.data_ptr(), wr.data_ptr(), eps, 1, spec.D, spec.E, x.data_ptr(), lg.data_ptr(), st)
    y2 = plain_forward(bm, L, x, lg, top_k, ws, kern)   # the block runs on the kernel without clusters too
    torch.cuda.synchronize()
    for rep in range(3):   # the same workspace, repeatedly
        h = h0.clone()
        bm.bitsmoe_moe_block_forward(h.data_ptr(), wr.data_ptr(), eps, 1, top_k, L, ws.ptr, ws.nbytes, st)
        torch.cuda.synchronize()
        assert bm.bitsmoe_last_device_status(ws.ptr) == 0
        two_step = (h0 + y2).cpu().numpy().astype(np.float64)   # the same fp32 add as the kernel's
        ymax, hmax = float(y2.abs().max()), float(h0.abs().max())
        assert np.max(np.abs(h.cpu().numpy() - two_step)) <= 1e-5 * ymax + 2.4e-7 * hmax
        upd = (h - h0).cpu().numpy().astype(np.float64)
    xo = x.cpu().numpy().view(np.uint16)
    ref = oracle.moe_forward_factored(layer, xo, lg.cpu().numpy().astype(np.float64), top_k)
    assert rel_err(upd, ref) <= TOL


@pytest.mark.parametrize("T", [2, 3, 4])
def test_few_tokens_as_fused_forwards(env, T):
    """Two to four tokens run as one fused forward per token on one workspace: plain and
    as a pre-norm block (norm mode), against the oracle and the two-step path."""
    torch, bm, kern = env
    spec = small(E=8, top_k=3, n=72)
    layer = synth.make_layer(spec, seed=30 + T, alpha_scale=3.0)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_forward_launches(L, T, spec.top_k) == T
    assert bm.bitsmoe_forward_plan(L, T, spec.top_k) == bm.PLAN_FUSED | (
        bm.PLAN_CLUSTERED if kern == "clustered" else 0)
    x, logits = synth.make_inputs(spec, T, seed=30 + T)
    ws = bm.Workspace(L, T, spec.top_k)
    y = bm.moe_forward(L, torch.from_numpy(x.view(np.int16)).cuda(), torch.from_numpy(logits).cuda(), spec.top_k,
                       ws=ws)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL
    # pre-norm block: h += MoE(RMSNorm(h)) token by token in the fused kernels
    wr = torch.from_numpy(synth.make_router_weight(spec, seed=30 + T).view(np.int16)).cuda()
    h0 = torch.from_numpy(synth.make_hidden(spec, T, seed=30 + T)).cuda()
    st = torch.cuda.current_stream().cuda_stream
    xb = torch.empty((T, spec.D), dtype=torch.int16, device="cuda")
    lg = torch.empty((T, spec.E), dtype=torch.float32, device="cuda")
    bm.bitsmoe_rmsnorm_router(h0.data_ptr(), wr.data_ptr(), 1e-6, T, spec.D, spec.E, xb.data_ptr(), lg.data_ptr(), st)
    y2 = plain_forward(bm, L, xb, lg, spec.top_k, ws, kern)
    h = h0.clone()
    bm.bitsmoe_moe_block_forward(h.data_ptr(), wr.data_ptr(), 1e-6, T, spec.top_k, L, ws.ptr, ws.nbytes, st)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    two_step = (h0 + y2).cpu().numpy().astype(np.float64)
    ymax, hmax = float(y2.abs().max()), float(h0.abs().max())
    assert np.max(np.abs(h.cpu().numpy() - two_step)) <= 1e-5 * ymax + 2.4e-7 * hmax


def test_bounded_wait_runs_out_and_is_reported(env):
    """Block 0 skips its arrival at the first grid barrier (testing hook) and every wait is
    bounded to about a millisecond: the kernel returns, the status word reports TIMEOUT (no
    trap, the context stays usable), and the next call on the same workspace is correct."""
    torch, bm, kern = env
    spec = small(E=8, top_k=2, n=72)
    layer = synth.make_layer(spec, seed=40)
    L = bm.bitsmoe_pack(layer, device=0)
    ws = bm.Workspace(L, 1, spec.top_k)
    x, logits = synth.make_inputs(spec, 1, seed=40)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ld = torch.from_numpy(logits).cuda()
    bm.bitsmoe_debug_wait_limit(1, 2_000_000)
    try:
        bm.moe_forward(L, xd, ld, spec.top_k, ws=ws)
        torch.cuda.synchronize()
    finally:
        bm.bitsmoe_debug_wait_limit(0, 0)
    assert bm.bitsmoe_last_device_status(ws.ptr) == bm.ERR_CODE["TIMEOUT"]
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0          # read and cleared
    check(env, layer, x, logits, spec.top_k, L=L, ws=ws)       # the next call's counters were cleared


def test_debug_bounds_check_reports_and_skips(env):
    """Debug bounds mode (the stand-in for a memory checker): the gate/up staging records of
    the token's first-ranked expert are shifted by the image's size, past its end.  The layer
    was loaded in that mode, so a zero-filled slack of the image's own size follows it, and the
    shifted copies would read mapped zeros even if a check were missing.  The kernel reports
    BITSMOE_ERR_DEVICE_BOUNDS and returns; with the records shifted back the next call on the
    same workspace matches the oracle."""
    torch, bm, kern = env
    spec = small(E=8, top_k=2, n=72)
    layer = synth.make_layer(spec, seed=45)
    bm.bitsmoe_debug_bounds(1)
    try:
        L = bm.bitsmoe_pack(layer, device=0)
        img = int(L.bytes()["total"])
        ws = bm.Workspace(L, 1, spec.top_k)
        x, logits = synth.make_inputs(spec, 1, seed=45)
        e = int(np.argmax(logits[0]))
        check(env, layer, x, logits, spec.top_k, L=L, ws=ws)       # in bounds: no report
        assert bm.bitsmoe_last_device_status(ws.ptr) == 0
        bm.bitsmoe_debug_shift_expert_records(L, e, img)
        xd = torch.from_numpy(x.view(np.int16)).cuda()
        ld = torch.from_numpy(logits).cuda()
        bm.moe_forward(L, xd, ld, spec.top_k, ws=ws)
        torch.cuda.synchronize()
        assert bm.bitsmoe_last_device_status(ws.ptr) == bm.ERR_CODE["DEVICE_BOUNDS"]
        bm.bitsmoe_debug_shift_expert_records(L, e, -img)
        check(env, layer, x, logits, spec.top_k, L=L, ws=ws)
        assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    finally:
        bm.bitsmoe_debug_bounds(0)


def test_clustered_plan_for_qw3_dims(env):
    """The Qwen3-shaped layer (full dims, top-8) runs on the clustered kernel at one token when
    it is forced (the device holds a cluster per (routing slot, row block) pair) and on the
    other one; both match the oracle."""
    torch, bm, kern = env
    spec = synth.scaled_spec(synth.WORKLOADS["qw3"], E=16, top_k=8)
    layer = synth.make_layer(spec, seed=41)
    L = bm.bitsmoe_pack(layer, device=0)
    plan = bm.bitsmoe_forward_plan(L, 1, 8)
    assert plan == bm.PLAN_FUSED | (bm.PLAN_CLUSTERED if kern == "clustered" else 0), plan
    for step in range(2):
        x, logits = synth.make_inputs(spec, 1, seed=41, step=step)
        check(env, layer, x, logits, 8, L=L)
