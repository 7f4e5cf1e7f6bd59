"""Transform from the model weights (Sec. 5 Step 1, Eq. AB-factorization; Appendix Proposition).

The oracle follows the paper's steps (Cholesky of Sigma_X, SVD of the whitened weight); these
pins tie it to identities the paper states and to independent computations, and the library's
planner (an eigen-decomposition of K^T K / n, no Cholesky) is checked against it."""
import math

import numpy as np
import pytest

from oracle import aatc_oracle as O
import workloads as W

SEED = 1002


def _case(d_model=256, n=4096, kind=0, head=0):
    x = W.hidden_states(SEED, 0, d_model, n).astype(np.float64)
    w = W.projection_weight(SEED, 0, kind, d_model, head + 1)[:, head * 128:(head + 1) * 128].astype(np.float64)
    return x, w


def test_factorization_reproduces_the_projection():
    """Eq. AB-factorization: W = L^-T U S P^T = A B."""
    x, w = _case()
    r = O.whitening_transform(x, w)
    np.testing.assert_allclose(r["A"] @ r["B"], w, rtol=0, atol=1e-11 * np.abs(w).max())


def test_cached_coefficients_are_decorrelated_with_variances_s():
    """Sec. 5 Step 1: S = A^T Sigma_X A, i.e. H = X A has H^T H / T = diag(S) (read with the
    1/T of Sigma_X), decorrelated and ordered by S."""
    x, w = _case()
    r = O.whitening_transform(x, w)
    h = x @ r["A"]
    cov = h.T @ h / x.shape[0]
    np.testing.assert_allclose(cov, np.diag(r["S"]), rtol=0, atol=1e-9 * r["S"].max())
    assert np.all(np.diff(r["S"]) <= 0)


def test_proposition_right_singular_vectors_of_k():
    """Appendix Proposition (1): P equals the right singular vectors of K = X W, computed here by
    an SVD of K itself (a different matrix and route from the whitened weight)."""
    x, w = _case(d_model=192, n=3000)
    r = O.whitening_transform(x, w)
    _, s_k, vt = np.linalg.svd(x @ w, full_matrices=False)
    np.testing.assert_allclose(s_k / math.sqrt(x.shape[0]), r["S"], rtol=1e-9)
    np.testing.assert_allclose(O.canonical_sign(vt.T), r["P"], atol=1e-7)


def test_proposition_coordinates_with_symmetric_square_root():
    """Appendix Proposition (2): K P = X Sigma_X^-1/2 U' S with the SVD Sigma_X^1/2 W = U' S P^T of
    the symmetric square root (an eigen-decomposition of Sigma_X, not the Cholesky factor)."""
    x, w = _case(d_model=128, n=3000)
    sigma = x.T @ x / x.shape[0]
    lam, vec = np.linalg.eigh(sigma)
    root = vec @ np.diag(np.sqrt(lam)) @ vec.T
    inv_root = vec @ np.diag(1 / np.sqrt(lam)) @ vec.T
    u2, s2, pt2 = np.linalg.svd(root @ w, full_matrices=False)
    np.testing.assert_allclose(x @ w @ pt2.T, x @ inv_root @ u2 @ np.diag(s2), rtol=0,
                               atol=1e-9 * np.abs(x @ w).max())
    r = O.whitening_transform(x, w)
    np.testing.assert_allclose(s2, r["S"], rtol=1e-9)       # same singular values, Cholesky or symmetric root


def test_transform_equals_the_pca_basis_of_the_hot_path():
    """The hot path's basis is the eigenbasis of the key second moment (Sec. 3.1 KLT); for K = X W it
    is the transform's P, with eigenvalues S^2, and A sqrt(S) = W P."""
    x, w = _case()
    r = O.whitening_transform(x, w)
    lam, u = O.eigenbasis(O.second_moment(x @ w))
    np.testing.assert_allclose(lam, r["S"] ** 2, rtol=1e-9)
    np.testing.assert_allclose(u, r["P"], atol=1e-8)
    np.testing.assert_allclose(O.hidden_encode_operand(r["A"], r["S"]), w @ r["P"], rtol=0,
                               atol=1e-10 * np.abs(w).max())


def test_a_wrong_factor_breaks_the_pins():
    """A plausible slip (L instead of L^T in the whitened weight) fails the factorization pin."""
    x, w = _case(d_model=128, n=2000)
    sigma = x.T @ x / x.shape[0]
    l_chol = np.linalg.cholesky(sigma)
    u, s, pt = np.linalg.svd(l_chol @ w, full_matrices=False)
    a_bad = np.linalg.solve(l_chol.T, u) * np.sqrt(s)[None, :]
    b_bad = np.sqrt(s)[:, None] * pt
    assert np.abs(a_bad @ b_bad - w).max() > 1e-3 * np.abs(w).max()


# --- the library's planner against the oracle ----------------------------------------------------

@pytest.mark.parametrize("d_model,kind", [(128, 0), (256, 1), (384, 0)])
def test_planner_transform_matches_oracle(d_model, kind):
    import paper_2608_14191_gb300 as aatc
    x, w = _case(d_model=d_model, n=3000, kind=kind)
    r = O.whitening_transform(x, w)
    g = aatc.whitening_transform(x.astype(np.float32), w.astype(np.float32))
    # The planner squares (K^T K): an eigenvalue's error is ~ eps lam_max, so small singular
    # values are accurate relative to S_max, not to themselves.
    np.testing.assert_allclose(g["S"], r["S"], rtol=1e-7, atol=1e-9 * r["S"].max())
    np.testing.assert_allclose(g["P"], r["P"], atol=2e-5)
    np.testing.assert_allclose(g["B"], r["B"], atol=2e-5 * np.abs(r["B"]).max())
    np.testing.assert_allclose(g["A"], r["A"], atol=2e-5 * np.abs(r["A"]).max())
    np.testing.assert_allclose(g["A_hat"], w @ r["P"], atol=2e-5 * np.abs(w).max())


def test_planner_rejects_rank_deficient_weights():
    import paper_2608_14191_gb300 as aatc
    x, w = _case(d_model=128, n=2000)
    w = w.copy()
    w[:, 5] = w[:, 7]                                        # two equal columns: W~ loses rank
    with pytest.raises(aatc.AatcError):
        aatc.whitening_transform(x.astype(np.float32), w.astype(np.float32))


def test_hidden_operand_is_w_times_basis_in_bf16():
    import paper_2608_14191_gb300 as aatc
    import torch
    rng = np.random.default_rng(3)
    L, H, dm = 1, 2, 128
    wk = rng.standard_normal((L, dm, H * 128)).astype(np.float32)
    wv = rng.standard_normal((L, dm, H * 128)).astype(np.float32)
    basis = np.stack([np.linalg.qr(rng.standard_normal((128, 128)))[0] for _ in range(L * H * 2)])
    basis = basis.reshape(L, H, 2, 128, 128).astype(np.float32)
    out = aatc.hidden_operand(aatc.dims(L, H, H * 4), wk, wv, basis)
    got = torch.from_numpy(out.view(np.int16)).view(torch.bfloat16).float().numpy()
    for h in range(H):
        for kind, wl in ((0, wk), (1, wv)):
            ref = (wl[0][:, h * 128:(h + 1) * 128].astype(np.float64) @ basis[0, h, kind].astype(np.float64)).T
            ref_bf16 = torch.from_numpy(ref.astype(np.float32)).to(torch.bfloat16).float().numpy()
            np.testing.assert_array_equal(got[0, h, kind], ref_bf16)
