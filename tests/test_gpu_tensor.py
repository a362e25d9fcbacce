"""GPU parity of the multi-token path (T > 8): multi-block router, tensor-core
projections (tcgen05, split-K), staged gate/up and down kernels with token
batches, against the fp64 oracle.

Covers token counts at and around the MMA granularity (16), a count whose
tokens span two launches of the projections (more than 256), ragged D and n
(partial TMA boxes, rows beyond the basis), every bit-width and the output
basis accumulating into a residual.  Bar: max|y_gpu - y_ref| / ||y_ref||_inf
<= 2e-3.
"""
import numpy as np
import pytest

import oracle
import synth

pytestmark = pytest.mark.gpu
TOL = 2e-3
ALL_BITS = {0: 0.1, 1: 0.15, 2: 0.2, 3: 0.15, 4: 0.1, 6: 0.1, 8: 0.1, 16: 0.1}


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


@pytest.fixture(scope="module")
def small_layer(env):
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=100, E=8, I=256, n=75, group=64, top_k=3)
    layer = synth.make_layer(spec, seed=71, bits_dist=ALL_BITS, alpha_scale=4.0)
    return spec, layer, bm.bitsmoe_pack(layer, device=0)


@pytest.mark.parametrize("T", [9, 16, 17, 64, 300])
def test_tensor_path_token_counts(env, small_layer, T):
    torch, bm = env
    spec, layer, L = small_layer
    assert bm.bitsmoe_forward_launches(L, T, spec.top_k) == 5   # 16-bit units: the dp2a expert kernels
    assert bm.bitsmoe_forward_plan(L, T, spec.top_k) == bm.PLAN_TC_PROJECTIONS   # 16-bit units: dp2a gate/up
    x, logits = synth.make_inputs(spec, T, seed=T)
    y = bm.moe_forward(L, torch.from_numpy(x.view(np.int16)).cuda(), torch.from_numpy(logits).cuda(), spec.top_k)
    torch.cuda.synchronize()
    ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL


TC_BITS = {0: 0.1, 1: 0.15, 2: 0.2, 3: 0.15, 4: 0.15, 6: 0.15, 8: 0.1}


@pytest.mark.parametrize("T,E,k,D,n,I,group", [
    (9, 8, 3, 100, 75, 256, 128),     # ragged n: the last K-block is partly padding
    (33, 8, 2, 256, 200, 384, 128),   # several slot ranges per block, three row blocks
    (130, 4, 2, 96, 72, 512, 256),    # group of two row blocks
    (600, 4, 2, 64, 40, 256, 128),    # experts with more than 256 tokens: two token tiles
])
def test_tensor_expert_factors(env, T, E, k, D, n, I, group):
    """Gate/up and down factors on tcgen05 (codes as fp16 bit patterns, decoded once per
    row block; gate/up: scale * alpha * z as an fp16 pair with SiLU(gate) * up in the
    epilogue; down: h as an fp16 pair, group scales applied to the per-row-block partial
    sums): every bit-width below 16, token tiles split at 32 tokens."""
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=D, E=E, I=I, n=n, group=group, top_k=k)
    layer = synth.make_layer(spec, seed=T + n, bits_dist=TC_BITS, alpha_scale=4.0)
    L = bm.bitsmoe_pack(layer, device=0)
    assert bm.bitsmoe_forward_plan(L, T, k) == bm.PLAN_TC_PROJECTIONS | bm.PLAN_TC_GATE_UP | bm.PLAN_TC_DOWN
    x, logits = synth.make_inputs(spec, T, seed=T)
    ws = bm.Workspace(L, T, k)
    y = bm.moe_forward(L, torch.from_numpy(x.view(np.int16)).cuda(), torch.from_numpy(logits).cuda(), k, ws=ws)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    ref = oracle.moe_forward_factored(layer, x, logits, k)
    assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL


def test_tensor_experts_skewed_load(env):
    """One expert holding every token (a biased logit sends all tokens to expert 0) next
    to experts with a single token: full and partial token tiles in one call."""
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=128, E=8, I=384, n=120, group=128, top_k=2)
    layer = synth.make_layer(spec, seed=81, bits_dist=TC_BITS, alpha_scale=4.0)
    L = bm.bitsmoe_pack(layer, device=0)
    T = 24
    x, logits = synth.make_inputs(spec, T, seed=81)
    logits[:, 0] += 20.0
    y = bm.moe_forward(L, torch.from_numpy(x.view(np.int16)).cuda(), torch.from_numpy(logits).cuda(), 2)
    torch.cuda.synchronize()
    ref = oracle.moe_forward_factored(layer, x, logits, 2)
    assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL


def test_tensor_path_qw3_dims_ragged_tokens(env):
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["qw3"], E=16, top_k=4)
    layer = synth.make_layer(spec, seed=72)
    L = bm.bitsmoe_pack(layer, device=0)
    T = 40
    assert bm.bitsmoe_forward_plan(L, T, spec.top_k) == bm.PLAN_TC_PROJECTIONS | bm.PLAN_TC_GATE_UP | bm.PLAN_TC_DOWN
    x, logits = synth.make_inputs(spec, T, seed=72)
    y = bm.moe_forward(L, torch.from_numpy(x.view(np.int16)).cuda(), torch.from_numpy(logits).cuda(), spec.top_k)
    torch.cuda.synchronize()
    ref = oracle.moe_forward_factored(layer, x, logits, spec.top_k)
    assert rel_err(y.cpu().numpy().astype(np.float64), ref) <= TOL


def test_tensor_path_block_residual(env):
    """Stack block at 24 tokens: RMSNorm + router + MoE, y accumulated into h.
    Layer-local parity: the oracle's MoE is fed the GPU's own normalised x and
    logits (checked close to the oracle's), so near-tied routing cannot differ."""
    torch, bm = env
    spec = synth.scaled_spec(synth.WORKLOADS["tiny"], D=96, E=8, I=256, n=72, group=64, top_k=3)
    layer = synth.make_layer(spec, seed=73, bits_dist=ALL_BITS, alpha_scale=4.0)
    L = bm.bitsmoe_pack(layer, device=0)
    T, eps = 24, 1e-6
    h0 = synth.make_hidden(spec, T, seed=5)
    wr = synth.make_router_weight(spec, seed=5)
    wr_d = torch.from_numpy(wr.view(np.int16)).cuda()
    stream = torch.cuda.current_stream().cuda_stream
    # the block's own normalised activations and logits
    hd = torch.from_numpy(h0.copy()).cuda()
    xg = torch.empty((T, spec.D), dtype=torch.int16, device="cuda")
    lg = torch.empty((T, spec.E), dtype=torch.float32, device="cuda")
    bm.bitsmoe_rmsnorm_router(hd.data_ptr(), wr_d.data_ptr(), eps, T, spec.D, spec.E, xg.data_ptr(), lg.data_ptr(),
                              stream)
    ws = bm.Workspace(L, T, spec.top_k)
    bm.bitsmoe_moe_block_forward(hd.data_ptr(), wr_d.data_ptr(), eps, T, spec.top_k, L, ws.ptr, ws.nbytes, stream)
    torch.cuda.synchronize()
    assert bm.bitsmoe_last_device_status(ws.ptr) == 0
    x_bits = xg.cpu().numpy().view(np.uint16)
    logits = lg.cpu().numpy()
    x_ref = oracle.rms_norm(h0.astype(np.float64), eps)
    assert np.max(np.abs(oracle.bf16_bits_to_f64(x_bits) - x_ref)) <= 2.0 ** -7 * np.max(np.abs(x_ref))
    lref = oracle.router_logits(wr, x_bits)
    assert np.max(np.abs(logits - lref)) <= 1e-4 * np.max(np.abs(lref))
    delta_ref = oracle.moe_forward_factored(layer, x_bits, logits, spec.top_k)
    delta = hd.cpu().numpy().astype(np.float64) - h0.astype(np.float64)
    assert rel_err(delta, delta_ref) <= TOL
