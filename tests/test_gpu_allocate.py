"""GPU parity of the bit allocation (bitsmoe_allocate_bits, through the C ABI) against
the allocation oracle (oracle/allocator.py).

The allocation is integer work decided by fp32 costs computed in the same steps on both
sides, so the bar is bit-exact: every unit's bit-width must equal the oracle's, on ragged
unit counts, unit lengths that are not a multiple of 4, the exact gammas 0, 1/2 and 1,
budgets from 0 to more than every unit can use, duplicated units (ties between units)
and all-zero units.  For other gammas (powf on the device) the allocation must be
feasible and as good as the oracle's to within rounding.
"""
import os

import numpy as np
import pytest

import synth
from oracle import allocator as A

pytestmark = pytest.mark.gpu
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _kappa():
    out = {}
    with open(os.path.join(GOLDEN, "kappa_values.txt")) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                k, v = line.split()
                out[int(k)] = float(v)
    return out


KAPPA = _kappa()
KAPPA3 = np.array([KAPPA[2], KAPPA[3], KAPPA[4]], np.float32)


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


def _inputs(U, d, seed, n=2048):
    P, _ = synth.make_float_units(U, d, seed=seed)
    rng = np.random.default_rng([seed, 5])
    alpha = ((np.arange(U) % n) + 1.0) ** -0.5
    beta = rng.lognormal(0.0, 1.0, U)
    return P, alpha.astype(np.float32), beta.astype(np.float32)


def gpu_alloc(env, P, alpha, beta, gamma, budget, profile=False):
    torch, bm = env
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    pd, ad, bd = t(P.astype(np.float32)), t(alpha), t(beta)
    U, d = P.shape
    bits = torch.empty(U, dtype=torch.uint8, device="cuda")
    nb = bm.bitsmoe_allocate_workspace_bytes(U)
    ws = torch.empty(nb + 256, dtype=torch.uint8, device="cuda")
    ms = bm.bitsmoe_allocate_bits(pd.data_ptr(), ad.data_ptr(), bd.data_ptr(), gamma, U, d, KAPPA3, budget,
                                  bits.data_ptr(), (ws.data_ptr() + 255) // 256 * 256, nb,
                                  torch.cuda.current_stream().cuda_stream, profile=profile)
    torch.cuda.synchronize()
    return bits.cpu().numpy(), ms


def oracle_alloc(P, alpha, beta, gamma, budget):
    return A.allocate(A.costs(P, alpha, beta, gamma, KAPPA), budget)


def assert_same(got, want):
    if not np.array_equal(got, want):
        bad = np.nonzero(got != want)[0]
        raise AssertionError(f"{bad.size} units differ, first {bad[:5].tolist()}: "
                             f"{got[bad[:5]].tolist()} != {want[bad[:5]].tolist()}")


@pytest.mark.parametrize("U,d,gamma,per_unit,seed", [
    (37, 256, 1.0, 1.6, 0),       # ragged unit count
    (5000, 768, 0.5, 1.67, 1),    # Qwen3-shaped units, the paper's 2-bit budget per unit
    (20000, 512, 0.0, 2.0, 2),
    (3001, 100, 1.0, 3.0, 3),     # unit length not a multiple of 4 (scalar loads)
    (777, 768, 0.5, 0.3, 4),      # scarce bits: most units evicted
])
def test_allocation_matches_oracle_bit_exactly(env, U, d, gamma, per_unit, seed):
    P, alpha, beta = _inputs(U, d, seed)
    budget = int(per_unit * U)
    got, _ = gpu_alloc(env, P, alpha, beta, gamma, budget)
    want = oracle_alloc(P, alpha, beta, gamma, budget)
    assert_same(got, want)
    assert int(got.astype(np.int64).sum()) <= budget


@pytest.mark.parametrize("budget", [0, 1, 7, 10 ** 9])
def test_budget_extremes(env, budget):
    P, alpha, beta = _inputs(300, 256, 7)
    got, _ = gpu_alloc(env, P, alpha, beta, 1.0, budget)
    assert_same(got, oracle_alloc(P, alpha, beta, 1.0, budget))
    if budget == 0:
        assert not got.any()


def test_duplicated_and_zero_units(env):
    """Identical units tie on every efficiency (the lower unit index goes first); all-zero
    units have zero high-bit distortion."""
    P, alpha, beta = _inputs(400, 256, 8)
    P[200:] = P[:200]
    alpha[200:] = alpha[:200]
    beta[200:] = beta[:200]
    P[10] = 0.0
    P[11] = 0.0
    for budget in (150, 333, 641, 1200):
        got, _ = gpu_alloc(env, P, alpha, beta, 0.5, budget)
        assert_same(got, oracle_alloc(P, alpha, beta, 0.5, budget))


def test_larger_allocation_and_profile(env):
    """65536 Qwen3-shaped units (a quarter of a projection) with the profiling entry point."""
    P, alpha, beta = _inputs(65536, 768, 9)
    budget = int(1.67 * 65536)
    got, ms = gpu_alloc(env, P, alpha, beta, 0.5, budget, profile=True)
    assert len(ms) == 3 and all(m > 0 for m in ms)
    assert_same(got, oracle_alloc(P, alpha, beta, 0.5, budget))


def test_general_gamma_is_feasible_and_as_good(env):
    P, alpha, beta = _inputs(4000, 256, 10)
    budget = int(1.8 * 4000)
    got, _ = gpu_alloc(env, P, alpha, beta, 0.7, budget)
    assert int(got.astype(np.int64).sum()) <= budget
    w = (alpha * alpha) * np.power(beta, np.float32(0.7), dtype=np.float32)
    C = w[:, None] * A.distortion(P, KAPPA)
    want = A.allocate(C, budget)
    assert A.total_cost(C, got) == pytest.approx(A.total_cost(C, want), rel=1e-5)


def test_empty_call_is_a_no_op(env):
    torch, bm = env
    assert bm.bitsmoe_allocate_bits(0, 0, 0, 0.5, 0, 16, KAPPA3, 10, 0, 0, 0, 0) is None
