"""Head-group bases (Sec. 5 Step 1, remark on multi-head attention): the oracle's group plan and
group decode, pinned against the per-head oracle, plain attention and transform-coding facts."""
import numpy as np

from oracle import aatc_oracle as O

D = O.D


def _correlated_heads(rng, g_h, n, shared=0.8):
    """g_h heads whose vectors share one latent component (fraction `shared` of the energy) plus
    head-specific parts, each with a power-law spectrum."""
    lam = np.arange(1, D + 1, dtype=np.float64) ** -1.5
    common = (rng.standard_normal((n, D)) * np.sqrt(lam)) @ np.linalg.qr(rng.standard_normal((D, D)))[0]
    heads = []
    for _ in range(g_h):
        own = (rng.standard_normal((n, D)) * np.sqrt(lam)) @ np.linalg.qr(rng.standard_normal((D, D)))[0]
        mix = np.linalg.qr(rng.standard_normal((D, D)))[0]
        heads.append(np.sqrt(shared) * common @ mix + np.sqrt(1.0 - shared) * own)
    return np.stack(heads)                                          # (g_h, n, 128)


def test_one_head_group_is_the_per_head_plan_and_decode():
    rng = np.random.default_rng(1)
    x = _correlated_heads(rng, 1, 2048)[0]
    qs = [rng.standard_normal((512, D)) for _ in range(4)]
    p1 = O.plan_stream(x, 2.75, queries_by_head=qs)
    pg = O.plan_head_group(x[None], 2.75, queries_by_head=qs, group=4)
    np.testing.assert_array_equal(pg["bits"], p1["bits"])
    np.testing.assert_allclose(pg["basis"], p1["basis"], rtol=0, atol=1e-12)
    np.testing.assert_allclose(pg["scales"], p1["scales"], rtol=1e-12)
    k, v = rng.standard_normal((300, D)), rng.standard_normal((300, D))
    q = rng.standard_normal((4, D))
    hk, hv = k @ p1["basis"], v @ p1["basis"]
    ref = O.decode_attention(q, hk[None], hv[None], p1["basis"][None], p1["basis"][None], 4)
    got = O.decode_attention_head_group(q, hk, hv, p1["basis"], p1["basis"], 4)
    np.testing.assert_allclose(got, ref, rtol=1e-12, atol=1e-12)


def test_group_decode_with_exact_coefficients_is_plain_attention():
    """With h = k_group U (no quantization) the group decode equals softmax(q . k_m / sqrt(128)) v_m
    for every query head of kv-head m: the orthonormal group basis preserves each block's dot
    products."""
    rng = np.random.default_rng(2)
    g_h, group, n = 4, 3, 257
    xk = _correlated_heads(rng, g_h, 4096)
    xv = _correlated_heads(rng, g_h, 4096)
    pk = O.plan_head_group(xk, 3.0, queries_by_head=[rng.standard_normal((256, D)) for _ in range(g_h * group)],
                           group=group)
    pv = O.plan_head_group(xv, 3.0)
    k = _correlated_heads(rng, g_h, n)                              # (g_h, n, 128)
    v = _correlated_heads(rng, g_h, n)
    kg = np.concatenate(list(k), axis=1)
    vg = np.concatenate(list(v), axis=1)
    q = rng.standard_normal((g_h * group, D))
    got = O.decode_attention_head_group(q, kg @ pk["basis"], vg @ pv["basis"], pk["basis"], pv["basis"], group)
    for i in range(g_h * group):
        ref = O.attention(q[i], k[i // group], v[i // group])
        np.testing.assert_allclose(got[i], ref, rtol=1e-10, atol=1e-12)


def test_block_diagonal_second_moment_splits_into_per_head_bases():
    """Calibration tokens that each excite one head only give an exactly block-diagonal second
    moment: the group eigenvalues are the union of the heads' and every group eigenvector lives in
    one head's block."""
    rng = np.random.default_rng(3)
    g_h, n = 3, 1500
    scales = [1.0, 0.37, 2.9]                                       # distinct spectra: no cross-head ties
    heads = np.zeros((g_h, g_h * n, D))
    for m in range(g_h):
        lam = scales[m] * np.arange(1, D + 1, dtype=np.float64) ** -1.2
        heads[m, m * n:(m + 1) * n] = (rng.standard_normal((n, D)) * np.sqrt(lam)) @ \
            np.linalg.qr(rng.standard_normal((D, D)))[0]
    p = O.plan_head_group(heads, 2.0, weights="var")
    per_head = np.sort(np.concatenate([O.eigenbasis(O.second_moment(heads[m]))[0] for m in range(g_h)]))[::-1]
    np.testing.assert_allclose(np.sort(p["sigma2"])[::-1], per_head, rtol=1e-9, atol=1e-15)
    u = p["basis"]
    for c in range(u.shape[1]):
        energy = np.array([np.sum(u[D * m:D * (m + 1), c] ** 2) for m in range(g_h)])
        assert np.max(energy) > 1.0 - 1e-10, (c, energy)


def test_group_budget_order_and_scales():
    rng = np.random.default_rng(4)
    x = _correlated_heads(rng, 4, 4096)
    for bits in (1.5, 2.75, 4.0):
        p = O.plan_head_group(x, bits, queries_by_head=[rng.standard_normal((256, D)) for _ in range(16)], group=4)
        assert p["bits"].shape == (4 * D,)
        assert int(p["bits"].sum()) == int(round(bits * 4 * D))
        assert np.all(np.diff(p["bits"]) <= 0)                      # non-increasing in storage order
        assert np.all(p["scales"][p["bits"] > 0] > 0)
        assert np.all(np.diff(p["g"]) <= 0)


def test_joint_group_transform_beats_separate_heads_for_correlated_heads():
    """Transform-coding gain: for heads sharing most of their energy, one basis and one
    water-filling over the group give a lower weighted distortion sum g_c 4^-b_c than separate
    per-head plans with the same total bits (w = 1, so g is the coefficient variance)."""
    rng = np.random.default_rng(5)
    g_h = 4
    x = _correlated_heads(rng, g_h, 8192, shared=0.9)
    for avg in (2.0, 2.75):
        pg = O.plan_head_group(x, avg, weights="var")
        joint = O.allocation_objective(pg["g"], pg["bits"])
        sep = 0.0
        for m in range(g_h):
            ph = O.plan_stream(x[m], avg, weights="var")
            sep += O.allocation_objective(ph["g"], ph["bits"])
        assert joint < 0.8 * sep, (avg, joint, sep)


def test_group_quantized_decode_error_falls_with_bits():
    """Through the group quantizer (group-wide alpha) and dequantizer, the decode error against
    exact attention shrinks as the budget grows."""
    rng = np.random.default_rng(6)
    g_h, group = 2, 4
    xk = _correlated_heads(rng, g_h, 4096)
    xv = _correlated_heads(rng, g_h, 4096)
    qcal = [rng.standard_normal((256, D)) for _ in range(g_h * group)]
    k = _correlated_heads(rng, g_h, 400)
    v = _correlated_heads(rng, g_h, 400)
    kg, vg = np.concatenate(list(k), axis=1), np.concatenate(list(v), axis=1)
    q = rng.standard_normal((g_h * group, D))
    exact = np.stack([O.attention(q[i], k[i // group], v[i // group]) for i in range(g_h * group)])
    errs = []
    for bits in (1.5, 2.75, 4.0, 6.0):
        pk = O.plan_head_group(xk, bits, queries_by_head=qcal, group=group)
        pv = O.plan_head_group(xv, bits)
        hk_hat = []
        for p, x in ((pk, kg), (pv, vg)):
            codes, alpha, _ = O.encode_stream(x, p["basis"], p["bits"], p["scales"])
            assert alpha.shape == (x.shape[0],)                     # one scale per token for the group
            hk_hat.append(O.dequantize(codes, alpha, p["scales"], p["bits"]))
        got = O.decode_attention_head_group(q, hk_hat[0], hk_hat[1], pk["basis"], pv["basis"], group)
        # relative to the value scale (the exact outputs average many values and can be small)
        errs.append(np.linalg.norm(got - exact) / (np.sqrt(np.mean(vg * vg) * D) * np.sqrt(len(q))))
    assert all(b < a for a, b in zip(errs, errs[1:])), errs
    assert errs[-1] < 0.01, errs


def _distinct_spectra_heads(rng, g_h, n):
    """g_h heads with different spectral decays and scales and a shared component (no
    near-degenerate eigenvalues between heads), for comparing two eigen-solvers."""
    heads = []
    common = rng.standard_normal((n, D))
    for m in range(g_h):
        lam = (1.0 + 0.7 * m) * np.arange(1, D + 1, dtype=np.float64) ** -(1.2 + 0.17 * m)
        basis = np.linalg.qr(rng.standard_normal((D, D)))[0]
        own = (rng.standard_normal((n, D)) * np.sqrt(lam)) @ basis
        heads.append(own + 0.3 * (common * np.sqrt(lam)) @ np.linalg.qr(rng.standard_normal((D, D)))[0])
    return np.stack(heads).astype(np.float32)


def test_library_head_group_planner_matches_oracle(aatc):
    """aatc_calibrate_head_group against plan_head_group: bits exact, basis / scales to fp32
    rounding, sigma^2 and weights to fp64 rounding (keys with query weights, values var-only)."""
    rng = np.random.default_rng(7)
    g_h, group, n, nq = 4, 4, 2048, 512
    x = _distinct_spectra_heads(rng, g_h, n)
    aniso = np.exp(-np.arange(D) / 40.0)
    q = (rng.standard_normal((g_h * group, nq, D)) * aniso).astype(np.float32)
    for qq, var in ((q, False), (None, True)):
        lib = aatc.calibrate_head_group(x, qq, 2.75, group=group, var_only=var)
        ref = O.plan_head_group(x.astype(np.float64), 2.75, queries_by_head=None if qq is None else list(qq.astype(np.float64)),
                                group=group, weights="var" if var else "aatc")
        np.testing.assert_array_equal(lib["bits"].astype(np.int64), ref["bits"])
        np.testing.assert_allclose(lib["sigma2"], ref["sigma2"], rtol=1e-9, atol=1e-14)
        np.testing.assert_allclose(lib["weights"], ref["weights"], rtol=1e-9, atol=1e-14)
        np.testing.assert_allclose(lib["basis"], ref["basis"], rtol=0, atol=2e-6)
        np.testing.assert_allclose(lib["scales"], ref["scales"], rtol=2e-6)


def test_library_head_group_planner_up_to_16_bits(aatc):
    """Two kv-heads (256 channels) at 6 bits with b_max = 16: bits match the oracle exactly and the
    leading channels take more than 8 bits."""
    rng = np.random.default_rng(8)
    x = _distinct_spectra_heads(rng, 2, 1024)
    lib = aatc.calibrate_head_group(x, None, 6.0, b_max=16)
    ref = O.plan_head_group(x.astype(np.float64), 6.0, b_max=16)
    got = lib["bits"].astype(np.int64)
    np.testing.assert_array_equal(got, ref["bits"])
    assert got.sum() == 6 * 256 and 8 < got.max() <= 16


def test_library_head_group_planner_rejects_bad_arguments(aatc):
    x = np.zeros((2, 16, D), np.float32)
    import pytest
    with pytest.raises(aatc.AatcError):
        aatc.calibrate_head_group(x[:, :1], None, 2.0)                # n_calib < 2
    with pytest.raises(aatc.AatcError):
        aatc.calibrate_head_group(x, None, 2.0 + 1.0 / 1000)         # budget not an integer
    with pytest.raises(ValueError):
        aatc.calibrate_head_group(x, np.zeros((3, 4, D), np.float32), 2.0, group=2)   # wrong query count
