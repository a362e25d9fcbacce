"""GPU shared-basis decomposition (bitsmoe_shared_basis) and calibration Gram
(bitsmoe_calibration_gram) against the oracle (oracle/bitsmoe_oracle.py::shared_basis_decompose,
numpy SVD in fp64; oracle/calibration.py::activation_metric).

Singular vectors are unique only up to sign (and only for simple singular values), so the
comparisons are: singular values directly; basis columns and spectral vectors after aligning
each column's sign with the oracle's, on matrices built with well separated singular values;
on generic random matrices the properties that fix the decomposition at any size
(orthonormal basis, W_cat rebuilt from P diag(alpha) Phi^T, unit spectral vectors).

Tolerances: the Gram matrix and the Jacobi rotations are fp32 (relative rounding ~1e-7 per
operation, thousands of rotations deep): singular values to 2e-5 of the largest; a basis
vector moves by about the Gram's rounding error over its eigenvalue gap, which is >= 0.2 % of
the largest eigenvalue in the prescribed matrices, so basis columns, alpha (||W_e phi_k||) and
the spectral vectors to 2e-4 (of the largest alpha for alpha); the rebuilt W_cat to 2e-5
(Frobenius, relative)."""
import numpy as np
import pytest

import synth
from oracle import bitsmoe_oracle as oracle
from oracle import calibration as C

pytestmark = pytest.mark.gpu


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


def split_experts(Wcat, E, side):
    return np.split(Wcat, E, axis=0 if side == "in" else 1)


def prescribed(E, d, D, side, seed):
    """W_cat with singular values spread evenly over [1, 3] (gaps >= 2/n), random singular
    vectors."""
    rng = np.random.default_rng(seed)
    R = E * d
    n = min(R, D)
    U = np.linalg.qr(rng.standard_normal((R, n)))[0]
    V = np.linalg.qr(rng.standard_normal((D, n)))[0]
    s = np.linspace(3.0, 1.0, n)
    Wcat = (U * s) @ V.T if side == "in" else (V * s) @ U.T
    return split_experts(Wcat.astype(np.float32), E, side)


def run(env, W, side, max_sweeps=30):
    torch, bm = env
    Wt = torch.from_numpy(np.stack(W)).cuda()
    phi, sig, alpha, P, sweeps, status = bm.shared_basis(Wt, side, max_sweeps=max_sweeps)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    return (phi.cpu().numpy().astype(np.float64), sig.cpu().numpy().astype(np.float64),
            alpha.cpu().numpy().astype(np.float64), P.cpu().numpy().astype(np.float64), int(sweeps.item()))


@pytest.mark.parametrize("side", ["in", "out"])
@pytest.mark.parametrize("E,d,D", [(3, 40, 72), (2, 33, 65), (4, 64, 256), (2, 20, 64)])
def test_against_oracle_with_separated_values(env, side, E, d, D):
    W = prescribed(E, d, D, side, seed=E * 100 + D)
    phi, sig, alpha, P, sweeps = run(env, W, side)
    Phi_r, A_r, P_r = oracle.shared_basis_decompose(W, side)
    S_r = np.linalg.svd(np.concatenate([w.astype(np.float64) for w in W], axis=0 if side == "in" else 1),
                        compute_uv=False)
    n = min(E * d, D)
    assert phi.shape == (D, n) and sig.shape == (n,) and alpha.shape == (E, n) and P.shape == (E, n, d)
    assert sweeps >= 1
    assert np.max(np.abs(sig - S_r[:n])) <= 2e-5 * S_r[0]
    sgn = np.sign(np.sum(phi * Phi_r[:, :n], axis=0))
    assert np.all(sgn != 0)
    assert np.max(np.abs(phi * sgn - Phi_r[:, :n])) <= 2e-4
    assert np.max(np.abs(alpha - A_r[:, :n])) <= 2e-4 * np.max(A_r)
    for e in range(E):
        assert np.max(np.abs(P[e] * sgn[:, None] - P_r[e][:, :n].T)) <= 2e-4
    # each basis column's largest component is positive
    idx = np.argmax(np.abs(phi), axis=0)
    assert np.all(phi[idx, np.arange(n)] > 0)


@pytest.mark.parametrize("side", ["in", "out"])
@pytest.mark.parametrize("E,d,D", [(8, 48, 128), (5, 77, 300)])
def test_properties_on_random_weights(env, side, E, d, D):
    rng = np.random.default_rng(D + E)
    W = [rng.standard_normal((d, D) if side == "in" else (D, d)).astype(np.float32) for _ in range(E)]
    phi, sig, alpha, P, _ = run(env, W, side)
    n = min(E * d, D)
    Wcat = np.concatenate([w.astype(np.float64) for w in W], axis=0 if side == "in" else 1)
    S_r = np.linalg.svd(Wcat, compute_uv=False)
    assert np.max(np.abs(sig - S_r[:n])) <= 2e-5 * S_r[0]
    assert np.all(np.diff(sig) <= 0)
    assert np.max(np.abs(phi.T @ phi - np.eye(n))) <= 2e-5
    # W_cat rebuilt from the factors: P~_e = P_e^T diag(alpha_e) (d x n)
    Pt = np.concatenate([P[e].T * alpha[e][None, :] for e in range(E)], axis=0)   # (E d) x n
    rebuilt = Pt @ phi.T if side == "in" else phi @ Pt.T
    assert np.linalg.norm(rebuilt - Wcat) <= 2e-5 * np.linalg.norm(Wcat)
    norms = np.linalg.norm(P, axis=2)
    live = alpha > 0
    assert np.max(np.abs(norms[live] - 1.0)) <= 1e-5


def test_zero_expert_block(env):
    """An expert whose weights are all zero has alpha = 0 and P = 0 (P~_e / 1)."""
    W = prescribed(3, 16, 40, "in", seed=9)
    W[1] = np.zeros_like(W[1])
    phi, sig, alpha, P, _ = run(env, W, "in")
    assert np.all(alpha[1] == 0) and np.all(P[1] == 0)
    Phi_r, A_r, P_r = oracle.shared_basis_decompose(W, "in")
    assert np.max(np.abs(alpha - A_r)) <= 2e-5 * np.max(A_r)


def test_bad_arguments(env):
    torch, bm = env
    lib = bm._lib()
    assert lib.bitsmoe_decompose_workspace_bytes(2, 1, 1, 8) == 0
    with pytest.raises(bm.BitsMoEError):
        bm.shared_basis(torch.zeros((1, 4, 1), device="cuda"), "in")   # D = 1


@pytest.mark.parametrize("T,D,weighted", [(0, 40, True), (37, 72, True), (300, 260, False)])
def test_calibration_gram(env, T, D, weighted):
    torch, bm = env
    rng = np.random.default_rng(T + D)
    x = synth.f32_to_bf16_bits(rng.standard_normal((max(T, 1), D)).astype(np.float32))[:T]
    g = rng.random(T).astype(np.float32) if weighted else np.ones(T, dtype=np.float32)
    xd = torch.from_numpy(x.view(np.int16).copy()).cuda().reshape(T, D)
    gd = torch.from_numpy(g).cuda() if weighted else None
    H = bm.calibration_gram(xd, gd).cpu().numpy().astype(np.float64)
    ref = C.activation_metric(oracle.bf16_bits_to_f64(x).T, g.astype(np.float64)) if T else np.zeros((D, D))
    assert H.shape == (D, D)
    scale = max(np.max(np.abs(ref)), 1e-30)
    assert np.max(np.abs(H - ref)) <= 2e-6 * scale * max(1.0, np.sqrt(T) / 4)
    assert np.array_equal(H, H.T)
