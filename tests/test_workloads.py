"""The synthetic input recipe (the stand-in for the paper's Llama / Qwen caches and calibration
sets): per stream a Haar-random basis, a power-law spectrum i^-1.5, four key outlier coordinates
x8, bf16-exact values, seeded sub-streams (no GPU)."""
import numpy as np

import workloads as W

CFG = W.CONFIGS["llama_layer"]


def test_haar_basis_is_orthogonal_and_seeded():
    a = W.stream_model(CFG.seed, 0, 3, W.KIND_V).mix
    b = W.stream_model(CFG.seed, 0, 3, W.KIND_V).mix
    c = W.stream_model(CFG.seed, 0, 4, W.KIND_V).mix
    assert np.array_equal(a, b) and not np.allclose(a, c)
    u = a / np.sqrt(W.power_law())[None, :]
    np.testing.assert_allclose(u.T @ u, np.eye(W.D), atol=1e-12)


def test_population_spectrum_is_the_power_law():
    """Values: covariance mix mix^T = U diag(i^-1.5) U^T exactly.  Keys: the same, with the four
    outlier coordinates scaled by 8 (their variance by 64)."""
    mv = W.stream_model(CFG.seed, 0, 0, W.KIND_V)
    lam = np.sort(np.linalg.eigvalsh(mv.mix @ mv.mix.T))[::-1]
    np.testing.assert_allclose(lam, W.power_law(), rtol=1e-9, atol=1e-15)
    mk = W.stream_model(CFG.seed, 0, 0, W.KIND_K)
    assert len(mk.outliers) == 4 and len(set(mk.outliers.tolist())) == 4 and mk.gain == 8.0
    g = np.ones(W.D)
    g[mk.outliers] = 8.0
    cov_k = (g[:, None] * (mk.mix @ mk.mix.T)) * g[None, :]
    x = mk.transform(np.random.default_rng(0).standard_normal((200000, W.D)))
    emp = x.T @ x / x.shape[0]
    assert np.abs(np.diag(emp) / np.diag(cov_k) - 1).max() < 0.02


def test_calibration_and_data_are_bf16_exact_and_distinct():
    cal = W.calibration_vectors(CFG, 0, 2, W.KIND_K, n=512)
    assert cal.dtype == np.float32 and np.array_equal(W.to_bf16(cal), cal)
    assert np.array_equal(cal, W.calibration_vectors(CFG, 0, 2, W.KIND_K, n=512))
    k, v = W.kv_host(CFG, 0, 1, 512)
    assert np.array_equal(W.to_bf16(k), k) and np.array_equal(W.to_bf16(v), v)
    assert not np.allclose(k[0, :, 2], cal)                      # different sub-stream
    # the empirical second moment of 4096 calibration vectors tracks the population spectrum
    x = W.calibration_vectors(CFG, 0, 1, W.KIND_V).astype(np.float64)
    emp = np.sort(np.linalg.eigvalsh(x.T @ x / x.shape[0]))[::-1]
    assert np.abs(emp[:8] / W.power_law()[:8] - 1).max() < 0.1


def test_bf16_rounding_matches_torch_cast():
    """to_bf16 (round to nearest even on the float32 bit pattern) gives the same values as
    torch's float32 -> bfloat16 cast: random magnitudes over 2^+-86, exact ties both ways,
    signed zeros, subnormals and the largest finite bf16 values."""
    import torch
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(1 << 18) * np.exp(rng.uniform(-60, 60, 1 << 18))).astype(np.float32)
    ties = (np.arange(1, 4097, dtype=np.uint32) << 16 | 0x8000).view(np.float32)
    x = np.concatenate([x, ties, -ties, np.array([0.0, -0.0, 3.3895314e38, -3.3895314e38, 1e-40, -1e-40],
                                                 np.float32)])
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()
    assert np.array_equal(W.to_bf16(x).view(np.uint32), ref.view(np.uint32))
    assert W.to_bf16(x.reshape(-1, 2)).shape == (x.size // 2, 2)
