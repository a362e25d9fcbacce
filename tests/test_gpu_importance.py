"""GPU parity of bitsmoe_importance (the importance beta of every unit from calibration
tokens, the bit allocation's input) against the fp64 calibration oracle
(oracle/calibration.py::factor_importance), on float factors of ragged sizes (no dimension a
multiple of the 64-wide tiles), with tied logits and a token whose affinity underflows.

Tolerance: the kernels sum fp32 products (z over D terms, then squares over the tokens; the
down projection through SiLU and two contractions over n and I terms), so each beta is within
a few fp32 roundings of the fp64 value: max |beta_gpu - beta_ref| / max |beta_ref| <= 1e-4 per
(projection, expert)."""
import numpy as np
import pytest

import synth
from oracle import calibration as C

pytestmark = pytest.mark.gpu
TOL = 1e-4


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


def float_factors(D, n, E, I, seed):
    """Orthonormal bases, energies j^-1/2 with an expert-dependent scale, and unit-norm
    Gaussian spectral vectors: the shapes and scales of a decomposition's output."""
    rng = np.random.default_rng(seed)
    Phi = [np.linalg.qr(rng.standard_normal((D, n)))[0].astype(np.float32) for _ in range(3)]
    j = np.arange(1, n + 1, dtype=np.float64)
    alpha = [np.stack([(j ** -0.5) * (1.0 + 0.1 * e) for e in range(E)]).astype(np.float32) for _ in range(3)]
    P = []
    for h in range(3):
        f = rng.standard_normal((E, I, n))
        f /= np.linalg.norm(f, axis=1, keepdims=True)
        P.append(f.astype(np.float32))
    return Phi, alpha, P


@pytest.mark.parametrize("D,n,E,I,k,T", [(96, 80, 6, 200, 2, 70), (256, 256, 8, 384, 3, 130), (72, 40, 33, 136, 4, 9)])
def test_importance_matches_oracle(env, D, n, E, I, k, T):
    torch, bm = env
    Phi, alpha, P = float_factors(D, n, E, I, seed=D + E)
    rng = np.random.default_rng(T)
    x = synth.f32_to_bf16_bits(rng.standard_normal((T, D)).astype(np.float32))
    logits = rng.integers(-3, 4, size=(T, E)).astype(np.float32)      # many exact ties
    logits[0, :] = 0.0
    logits[0, 1] = 120.0     # token 0: the other selected experts' gate weights underflow to 0
    ref = C.factor_importance(Phi, alpha, [[P[h][e] for e in range(E)] for h in range(3)], x, logits, k)
    dev = torch.device("cuda")
    tx = torch.from_numpy(x.view(np.int16)).to(dev)
    tl = torch.from_numpy(logits).to(dev)
    basis = [torch.from_numpy(Phi[h]).to(dev) for h in range(2)]
    al = [torch.from_numpy(alpha[h]).to(dev) for h in range(2)]
    fac = [torch.from_numpy(P[h]).to(dev) for h in range(3)]
    beta = bm.importance(tx, tl, k, basis, al, fac).cpu().numpy().astype(np.float64)
    assert beta.shape == (3, E, n)
    for h in range(3):
        for e in range(E):
            scale = max(np.max(np.abs(ref[h, e])), 1e-30)
            err = np.max(np.abs(beta[h, e] - ref[h, e])) / scale
            assert err <= TOL, (h, e, err)
    assert np.all(beta >= 0)


def test_importance_no_tokens_and_bad_args(env):
    torch, bm = env
    D, n, E, I, k = 64, 32, 4, 64, 2
    Phi, alpha, P = float_factors(D, n, E, I, seed=3)
    dev = torch.device("cuda")
    basis = [torch.from_numpy(Phi[h]).to(dev) for h in range(2)]
    al = [torch.from_numpy(alpha[h]).to(dev) for h in range(2)]
    fac = [torch.from_numpy(P[h]).to(dev) for h in range(3)]
    x = torch.zeros((0, D), dtype=torch.int16, device=dev)
    lg = torch.zeros((0, E), dtype=torch.float32, device=dev)
    beta = bm.importance(x, lg, k, basis, al, fac)
    assert bool((beta == 0).all())
    with pytest.raises(bm.BitsMoEError):
        bm.importance(torch.zeros((3, D), dtype=torch.int16, device=dev), torch.zeros((3, E), device=dev),
                      E + 1, basis, al, fac)
