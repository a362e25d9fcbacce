"""bitsmoe_moe_forward_noalloc: the forward for callers that cannot allocate
device memory (their device memory belongs to another allocator, or
allocating would synchronise the device in the middle of a decode loop).

It must give the same result as bitsmoe_moe_forward with a caller-provided
workspace, on consecutive calls that share its built-in scratch, and reject a
batch whose workspace would not fit that scratch.  Collected last on purpose:
the check passes alone in a fresh process and after every other test.
"""
import ctypes

import numpy as np
import pytest

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


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


def test_noalloc_matches_workspace_forward_on_consecutive_calls(env):
    torch, bm = env
    lib = bm._lib()
    spec = synth.WORKLOADS["qw3_skew"]
    spec = synth.scaled_spec(spec, D=512, E=16, I=384, n=512, top_k=4)
    layer = synth.make_layer(spec, seed=3)
    L = bm.bitsmoe_pack(layer, device=0)
    stream = torch.cuda.current_stream().cuda_stream
    for call, T in enumerate((5, 3)):            # two calls in a row share the scratch
        x, logits = synth.make_inputs(spec, T, seed=3, step=call)
        xd = torch.from_numpy(x.view(np.int16)).cuda()
        ld = torch.from_numpy(logits).cuda()
        y_ref = bm.moe_forward(L, xd, ld, spec.top_k)
        y = torch.full((T, spec.D), float("nan"), dtype=torch.float32, device="cuda")
        rc = lib.bitsmoe_moe_forward_noalloc(xd.data_ptr(), ld.data_ptr(), T, spec.top_k, L.handle,
                                             y.data_ptr(), ctypes.c_void_p(stream))
        assert rc == 0, bm.bitsmoe_strerror(rc)
        torch.cuda.synchronize()
        err = _rel(y.cpu().numpy().astype(np.float64), y_ref.cpu().numpy().astype(np.float64))
        assert err <= TOL, (call, err)


def test_noalloc_rejects_batches_beyond_its_scratch(env):
    torch, bm = env
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=4)
    L = bm.bitsmoe_pack(layer, device=0)
    T = 1
    while bm.bitsmoe_workspace_bytes(L, T, spec.top_k) <= bm.NOALLOC_SCRATCH_BYTES:
        T *= 2
    x = torch.zeros((T, spec.D), dtype=torch.int16, device="cuda")
    lg = torch.zeros((T, spec.E), dtype=torch.float32, device="cuda")
    y = torch.zeros((T, spec.D), dtype=torch.float32, device="cuda")
    with pytest.raises(bm.BitsMoEError) as ei:
        bm.bitsmoe_moe_forward_noalloc(x.data_ptr(), lg.data_ptr(), T, spec.top_k, L, y.data_ptr(), 0)
    assert ei.value.code == bm.ERR_CODE["WORKSPACE_TOO_SMALL"]


def test_noalloc_status_word_is_readable(env):
    """The caller cannot name the scratch, so its device status comes through its own accessor:
    zero after calls that completed (and it stays cleared on a second read)."""
    torch, bm = env
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=5)
    L = bm.bitsmoe_pack(layer, device=0)
    x, logits = synth.make_inputs(spec, 1, seed=5)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ld = torch.from_numpy(logits).cuda()
    y = torch.zeros((1, spec.D), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    bm.bitsmoe_moe_forward_noalloc(xd.data_ptr(), ld.data_ptr(), 1, spec.top_k, L, y.data_ptr(), stream)
    assert bm.bitsmoe_noalloc_last_status(stream) == 0
    assert bm.bitsmoe_noalloc_last_status(stream) == 0


_CAPTURE_FIRST = r"""
import ctypes, sys
import numpy as np, torch
sys.path.insert(0, sys.argv[1])
import synth, paper_2606_00079_gb300 as bm
spec = synth.WORKLOADS["tiny"]
L = bm.bitsmoe_pack(synth.make_layer(spec, seed=6), device=0)
x = torch.zeros((1, spec.D), dtype=torch.int16, device="cuda")
lg = torch.zeros((1, spec.E), dtype=torch.float32, device="cuda")
y = torch.zeros((1, spec.D), dtype=torch.float32, device="cuda")
s = torch.cuda.Stream()
torch.cuda.synchronize()
rc = None
g = torch.cuda.CUDAGraph()
try:
    with torch.cuda.graph(g, stream=s):
        rc = bm._lib().bitsmoe_moe_forward_noalloc(x.data_ptr(), lg.data_ptr(), 1, spec.top_k, L.handle,
                                                   y.data_ptr(), ctypes.c_void_p(s.cuda_stream))
except Exception:
    pass
print("RC", rc)
"""


def test_noalloc_first_call_inside_capture_is_refused(env):
    """A fresh process whose first no-allocation call on the device comes inside a stream
    capture gets BITSMOE_ERR_INVALID_ARG (the scratch address must be looked up before)."""
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "-c", _CAPTURE_FIRST, root], capture_output=True, text=True, timeout=300)
    assert "RC -1" in r.stdout, (r.stdout, r.stderr[-2000:])


def test_noalloc_status_reports_a_timeout(env):
    """A no-allocation call whose bounded wait runs out (testing hook: block 0 skips its first
    grid-barrier arrival) reports TIMEOUT through the no-allocation status accessor, and the
    next call on the shared scratch is correct again."""
    torch, bm = env
    lib = bm._lib()
    spec = synth.WORKLOADS["tiny"]
    layer = synth.make_layer(spec, seed=7)
    L = bm.bitsmoe_pack(layer, device=0)
    x, logits = synth.make_inputs(spec, 1, seed=7)
    xd = torch.from_numpy(x.view(np.int16)).cuda()
    ld = torch.from_numpy(logits).cuda()
    y = torch.zeros((1, spec.D), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream().cuda_stream
    bm.bitsmoe_debug_wait_limit(1, 2_000_000)
    try:
        bm.bitsmoe_moe_forward_noalloc(xd.data_ptr(), ld.data_ptr(), 1, spec.top_k, L, y.data_ptr(), stream)
        torch.cuda.synchronize()
    finally:
        bm.bitsmoe_debug_wait_limit(0, 0)
    assert bm.bitsmoe_noalloc_last_status(stream) == bm.ERR_CODE["TIMEOUT"]
    y_ref = bm.moe_forward(L, xd, ld, spec.top_k)
    rc = lib.bitsmoe_moe_forward_noalloc(xd.data_ptr(), ld.data_ptr(), 1, spec.top_k, L.handle, y.data_ptr(),
                                         ctypes.c_void_p(stream))
    assert rc == 0
    torch.cuda.synchronize()
    assert bm.bitsmoe_noalloc_last_status(stream) == 0
    assert _rel(y.cpu().numpy().astype(np.float64), y_ref.cpu().numpy().astype(np.float64)) <= TOL
