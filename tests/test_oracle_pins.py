"""Pins of the CPU oracle against what the paper and the mathematics fix (no GPU).

Each test names the passage it follows.  The checks are chosen so that a dropped
term, a wrong sign, a swapped operand or a wrong constant in the oracle fails one
of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest

from oracle import aatc_oracle as O
import workloads as W

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


# --- (1) transform round trip (Sec. 3.1: orthonormal transform, exactly invertible) ---------

def test_basis_orthonormal_and_round_trip():
    cfg = W.CONFIGS["tiny"]
    x = W.calibration_vectors(cfg, 0, 0, W.KIND_K).astype(np.float64)
    plan = O.plan_stream(x, 2.75)
    u = plan["basis"]
    assert np.max(np.abs(u.T @ u - np.eye(O.D))) < 1e-12
    h = x @ u
    assert np.max(np.abs(h @ u.T - x)) < 1e-12 * np.max(np.abs(x)) * O.D


def test_quantizer_round_trip_with_unlimited_bits():
    """With many bits per channel the transform + quantizer reproduces x up to Delta/2 per
    coefficient (Sec. 3.1 and Def. uniform-quant)."""
    cfg = W.CONFIGS["tiny"]
    x = W.calibration_vectors(cfg, 0, 0, W.KIND_K).astype(np.float64)
    plan = O.plan_stream(x, 2.75)
    bits = np.full(O.D, 24)
    codes, alpha, _ = O.encode_stream(x[:256], plan["basis"], bits, plan["scales"])
    hhat = O.dequantize(codes, alpha, plan["scales"], bits)
    delta = 2 * alpha[:, None] * plan["scales"][None, :] / 2.0 ** 24
    h = x[:256] @ plan["basis"]
    # inside the range |x - xhat| <= Delta/2; the positive extreme clamps (error <= Delta)
    assert np.all(np.abs(hhat - h) <= delta + 1e-12 * np.abs(h))
    xhat = hhat @ plan["basis"].T
    assert np.max(np.abs(xhat - x[:256])) < 1e-5 * np.max(np.abs(x))


# --- (2) reverse water-filling closed form (Eq. bit-allocation) ------------------------------

@pytest.mark.parametrize("case", _gold("waterfill_textbook.json")["cases"])
def test_continuous_waterfilling_textbook(case):
    bits, theta = O.continuous_allocation(np.array(case["sigma2"]), case["budget"])
    assert theta == pytest.approx(case["theta"], rel=1e-9)
    np.testing.assert_allclose(bits, case["bits"], atol=1e-9)


def test_continuous_waterfilling_kkt():
    """Every active channel ends at the same distortion theta (Sec. 3.1: each retained
    coefficient is quantized to the same distortion c*lambda), inactive channels lie below the
    water level, and the budget is met."""
    rng = np.random.default_rng(5)
    g = np.exp(rng.normal(0, 3, 64))
    bits, theta = O.continuous_allocation(g, 64 * 1.5)
    assert np.sum(bits) == pytest.approx(64 * 1.5, rel=1e-9)
    act = bits > 0
    np.testing.assert_allclose(g[act] * 2.0 ** (-2 * bits[act]), theta, rtol=1e-9)
    assert np.all(g[~act] <= theta * (1 + 1e-9))


# --- (3) brute force at d = 4 (Eq. waterfilling-keys, integer widths) -----------------------

def test_greedy_matches_brute_force_d4():
    rng = np.random.default_rng(11)
    for trial in range(300):
        g = np.exp(rng.normal(0, 2.5, 4)) * rng.choice([1, 1, 0.01], 4)
        budget = int(rng.integers(0, 33))
        b_max = 8
        best = min(O.allocation_objective(g, b) for b in itertools.product(range(b_max + 1), repeat=4)
                   if sum(b) <= budget)
        got = O.greedy_allocation(g, budget, b_max)
        assert got.sum() <= budget and got.max() <= b_max and got.min() >= 0
        assert O.allocation_objective(g, got) == pytest.approx(best, rel=1e-12), (g, budget)


def test_greedy_matches_brute_force_d3_up_to_16_bits():
    """The paper's widths b in {0..16}: exhaustive search over 17^3 allocations at d = 3."""
    rng = np.random.default_rng(12)
    grid = np.array(list(itertools.product(range(17), repeat=3)))
    for trial in range(40):
        g = np.exp(rng.normal(0, 6, 3))
        budget = int(rng.integers(0, 49))
        ok = grid.sum(axis=1) <= budget
        best = np.min(np.sum(g[None, :] * 4.0 ** -grid[ok], axis=1))
        got = O.greedy_allocation(g, budget, 16)
        assert got.sum() == budget and got.max() <= 16
        assert O.allocation_objective(g, got) == pytest.approx(best, rel=1e-12), (g, budget)


def test_greedy_integer_local_optimality_and_monotone():
    """Exchange optimality of the integer allocation: moving one bit between any two channels
    never lowers the objective; with g sorted descending the widths are non-increasing."""
    rng = np.random.default_rng(3)
    g = np.sort(np.exp(rng.normal(0, 2, 128)))[::-1]
    for budget in (192, 256, 352, 512):
        b = O.greedy_allocation(g, budget, 8)
        assert b.sum() == budget
        assert np.all(np.diff(b) <= 0)
        base = O.allocation_objective(g, b)
        for i in range(128):
            for j in range(128):
                if i != j and b[i] > 0 and b[j] < 8:
                    bb = b.copy()
                    bb[i] -= 1
                    bb[j] += 1
                    assert O.allocation_objective(g, bb) >= base * (1 - 1e-12)


def test_greedy_saturates_at_b_max():
    """A budget of at least d b_max bits fills every channel to b_max and no further (widths in
    {0..b_max}, Eq. waterfilling-keys); a budget of d b_max - 1 leaves exactly the channel with
    the smallest g one bit short."""
    g = np.exp(np.random.default_rng(4).normal(0, 3, 16))
    for b_max in (1, 3, 8):
        np.testing.assert_array_equal(O.greedy_allocation(g, 16 * b_max + 40, b_max), np.full(16, b_max))
        short = O.greedy_allocation(g, 16 * b_max - 1, b_max)
        want = np.full(16, b_max)
        want[int(np.argmin(g))] -= 1
        np.testing.assert_array_equal(short, want)


# --- (4) Theorem 1: D ~= D_K + D_V under the white-noise model -------------------------------

def test_theorem1_monte_carlo():
    """Inject independent symmetric (uniform) noise into keys and values; the Monte Carlo
    output distortion approaches D_K + D_V as the noise shrinks (Theorem 1, remainder higher
    order in the noise scale)."""
    rng = np.random.default_rng(7)
    t, d = 24, 8
    q = rng.standard_normal(d) * 2.0
    k = rng.standard_normal((t, d))
    v = rng.standard_normal((t, d))
    wo = rng.standard_normal((d, 6)) / math.sqrt(d)
    o = O.attention(q, k, v, wo)
    ratios = []
    for eps in (0.3, 0.03):
        half_k = eps * rng.uniform(0.5, 1.5, (t, d))
        half_v = eps * rng.uniform(0.5, 1.5, (t, d))
        var_k, var_v = half_k ** 2 / 3, half_v ** 2 / 3
        dk, dv = O.distortion_decomposition(q, k, v, var_k, var_v, wo)
        n = 20000
        acc = 0.0
        for _ in range(n):
            kk = k + rng.uniform(-1, 1, (t, d)) * half_k
            vv = v + rng.uniform(-1, 1, (t, d)) * half_v
            acc += np.sum((O.attention(q, kk, vv, wo) - o) ** 2)
        ratios.append((acc / n) / (dk + dv))
        assert dk > 0.1 * dv and dv > 0.1 * dk        # both terms matter
    assert abs(ratios[1] - 1) < 0.04
    assert abs(ratios[1] - 1) < abs(ratios[0] - 1) + 0.02


def test_theorem1_value_term_exact_for_key_free_noise():
    """Without key noise the output error is linear in the value noise, so D = D_V exactly."""
    rng = np.random.default_rng(8)
    t, d = 10, 6
    q, k, v = rng.standard_normal(d), rng.standard_normal((t, d)), rng.standard_normal((t, d))
    var_v = rng.uniform(0.01, 0.1, (t, d))
    dk, dv = O.distortion_decomposition(q, k, v, np.zeros((t, d)), var_v)
    a = O.softmax(k @ q / math.sqrt(d))
    assert dk == 0.0
    assert dv == pytest.approx(float(np.sum(a[:, None] ** 2 * var_v)), rel=1e-12)


# --- Appendix Proposition: whitening-SVD transform == PCA of K = XW ---------------------------

def test_whitening_svd_equals_pca():
    rng = np.random.default_rng(2)
    n, dm, d = 5000, 48, 16
    x = rng.standard_normal((n, dm)) @ rng.standard_normal((dm, dm)) / math.sqrt(dm)
    w = rng.standard_normal((dm, d))
    sig_x = x.T @ x / n
    l_chol = np.linalg.cholesky(sig_x)
    _, s, pt = np.linalg.svd(l_chol.T @ w, full_matrices=False)
    lam, u = O.eigenbasis(O.second_moment(x @ w))
    np.testing.assert_allclose(lam, s ** 2, rtol=1e-9)
    np.testing.assert_allclose(u, O.canonical_sign(pt.T), atol=1e-8)


# --- basis-scaling invariance (derived from Eq. AB-factorization, Sec. 5) -----------------------

def test_allocation_and_codes_invariant_to_column_scaling():
    """Scaling encode column c by kappa_c (and the reconstruction row by 1/kappa_c) leaves
    g_c = w_c sigma_c^2, the widths and every code unchanged: sigma^2 and s use the encode
    basis A, w uses the reconstruction B."""
    cfg = W.CONFIGS["tiny"]
    x = W.calibration_vectors(cfg, 0, 0, W.KIND_K).astype(np.float64)
    qs = [W.calibration_queries(cfg, 0, j, anisotropic=True).astype(np.float64) for j in range(4)]
    plan = O.plan_stream(x, 2.75, queries_by_head=qs)
    u = plan["basis"]
    kappa = np.random.default_rng(4).uniform(0.2, 5.0, O.D)
    a2, b2 = u * kappa[None, :], (u * (1 / kappa)[None, :]).T
    g1 = O.key_weights(u.T, qs) * O.channel_variance(u, x)
    g2 = O.key_weights(b2, qs) * O.channel_variance(a2, x)
    np.testing.assert_allclose(g1, g2, rtol=1e-10)
    np.testing.assert_allclose(g1, plan["g"], rtol=1e-10)
    bits = plan["bits"]
    c1, _, _ = O.encode_stream(x[:500], u, bits, O.channel_scales(u, x))
    c2, _, _ = O.encode_stream(x[:500], a2, bits, O.channel_scales(a2, x))
    assert np.array_equal(c1, c2)


def test_key_weights_gqa_hand_example():
    """GQA weights sum the per-head mean squared projections (appendix GQA remark)."""
    b = np.array([[1.0, 0.0], [0.6, 0.8]])
    q1 = np.array([[1.0, 2.0], [3.0, 0.0]])
    q2 = np.array([[0.0, 1.0]])
    # head 1: channel 0: (1^2 + 3^2)/2 = 5; channel 1: (0.6+1.6)^2=4.84, (1.8)^2=3.24 -> 4.04
    # head 2: channel 0: 0; channel 1: 0.8^2 = 0.64
    np.testing.assert_allclose(O.key_weights(b, [q1, q2]), [5.0, 4.68], rtol=1e-12)
    np.testing.assert_allclose(O.value_weights(b), [1.0, 1.0], rtol=1e-12)
    np.testing.assert_allclose(O.value_weights(b, np.diag([2.0, 0.5])), [4.0, 0.36 * 4 + 0.64 * 0.25])


# --- quantizer (Def. uniform-quant; Sec. 5 symmetric quantizer; Eq. noise-model) ---------------

def test_quantizer_error_bound_and_clamp():
    rng = np.random.default_rng(9)
    s = np.ones(O.D)
    for b in (1, 2, 3, 5, 8, 12, 16):
        bits = np.full(O.D, b)
        h = rng.uniform(-1, 1, (400, O.D))
        alpha = O.token_scale(h, s, bits)
        codes, _ = O.quantize(h, alpha, s, bits)
        hhat = O.dequantize(codes, alpha, s, bits)
        delta = 2 * alpha[:, None] / 2.0 ** b
        assert codes.min() >= -2 ** (b - 1) and codes.max() <= 2 ** (b - 1) - 1
        top = codes == 2 ** (b - 1) - 1
        err = np.abs(h - hhat)
        # within range error <= Delta/2; at the clamped positive extreme error <= Delta (slack: the
        # fp64 rounding of h - h_hat, ~2^-52 |h|, with |h| up to 2^(b-1) Delta)
        slack = 1e-15 * np.abs(h)
        dd = delta.repeat(O.D, 1)
        assert np.all(err[~top] <= dd[~top] / 2 * (1 + 1e-12) + slack[~top])
        assert np.all(err <= dd * (1 + 1e-12) + slack)
        # the argmax coefficient sits exactly at +-2^(b-1) steps
        tmax = np.max(np.abs(h), axis=1) / delta[:, 0]
        np.testing.assert_allclose(tmax, 2.0 ** (b - 1), rtol=1e-12)


def test_quantizer_specific_values():
    """Hand cases of floor(h/Delta + 1/2) with Delta = 2 alpha s / 2^b (round half up)."""
    s = np.array([1.0, 1.0, 1.0, 1.0])
    bits = np.array([2, 2, 2, 2])
    h = np.array([[1.0, 0.25, -0.25, -0.75]])       # alpha = 1, Delta = 0.5
    codes, t = O.quantize(h, np.array([1.0]), s, bits)
    np.testing.assert_allclose(t, [[2.0, 0.5, -0.5, -1.5]])
    assert codes.tolist() == [[1, 1, 0, -1]]          # +2 clamps to 1; +-1/2 round up
    codes, _ = O.quantize(np.zeros((1, 4)), np.array([0.0]), s, bits)
    assert codes.tolist() == [[0, 0, 0, 0]]


def test_noise_model_high_rate():
    """E[dH^2] = Delta^2/12 at high rate (Eq. noise-model)."""
    rng = np.random.default_rng(10)
    b = 7
    s = np.ones(O.D)
    bits = np.full(O.D, b)
    h = rng.normal(0, 0.3, (4000, O.D))
    h[:, 0] = 1.0                                  # fixes alpha = 1
    codes, _ = O.quantize(h, O.token_scale(h, s, bits), s, bits)
    err = O.dequantize(codes, O.token_scale(h, s, bits), s, bits)[:, 1:] - h[:, 1:]
    delta = 2.0 / 2 ** b
    assert np.mean(err ** 2) == pytest.approx(delta ** 2 / 12, rel=0.03)


def test_token_scale_ignores_dropped_channels():
    h = np.array([[0.5, -2.0, 100.0]])
    s = np.array([1.0, 4.0, 1.0])
    assert O.token_scale(h, s, np.array([3, 2, 0]))[0] == pytest.approx(0.5)


def test_percentile_definition():
    assert O.percentile_linear(np.arange(101.0), 99) == 99.0
    assert O.percentile_linear(np.arange(11.0)[::-1], 99) == pytest.approx(9.9)
    assert O.percentile_linear(np.array([2.0, 0.0]), 50) == 1.0


def test_channel_scale_is_p99_of_magnitudes():
    """s_c is the 99th percentile of |h_c| over the calibration tokens (Sec. 5): with the identity
    basis and a column holding -100 .. 0 (magnitudes 0 .. 100, 101 samples) it is exactly 99; a
    column of +-1 gives 1; a scaled column scales s_c."""
    x = np.zeros((101, O.D))
    x[:, 0] = -np.arange(101.0)[::-1]
    x[:, 1] = np.where(np.arange(101) % 2 == 0, 1.0, -1.0)
    x[:, 2] = 0.5 * np.arange(101.0)
    s = O.channel_scales(np.eye(O.D), x)
    assert s[0] == pytest.approx(99.0, rel=1e-15)
    assert s[1] == 1.0
    assert s[2] == pytest.approx(49.5, rel=1e-15)
    assert np.all(s[3:] == 0.0)


# --- decode = SDPA over reconstructed keys and values (Alg. 1, Def. sdpa) ----------------------

def test_decode_matches_library_sdpa():
    import torch
    rng = np.random.default_rng(12)
    hkv, g, n = 2, 3, 50
    basis = np.stack([np.linalg.qr(rng.standard_normal((O.D, O.D)))[0] for _ in range(2 * hkv)])
    bk, bv = basis[:hkv], basis[hkv:]
    hk = rng.standard_normal((hkv, n, O.D))
    hv = rng.standard_normal((hkv, n, O.D))
    q = rng.standard_normal((hkv * g, O.D))
    out = O.decode_attention(q, hk, hv, bk, bv, g)
    for j in range(hkv * g):
        h = j // g
        kk = torch.from_numpy(hk[h] @ bk[h].T)[None, None]
        vv = torch.from_numpy(hv[h] @ bv[h].T)[None, None]
        ref = torch.nn.functional.scaled_dot_product_attention(torch.from_numpy(q[j])[None, None, None], kk, vv)
        np.testing.assert_allclose(out[j], ref.numpy().reshape(-1), rtol=1e-10, atol=1e-12)


def test_decode_special_cases():
    rng = np.random.default_rng(13)
    u = np.linalg.qr(rng.standard_normal((O.D, O.D)))[0]
    hv = rng.standard_normal((1, 5, O.D))
    # one token: the output is the reconstructed value
    out = O.decode_attention(rng.standard_normal((2, O.D)), rng.standard_normal((1, 1, O.D)),
                             hv[:, :1], u[None], u[None], 2)
    np.testing.assert_allclose(out[0], u @ hv[0, 0], atol=1e-12)
    # identical keys: uniform attention, the mean value
    hk = np.repeat(rng.standard_normal((1, 1, O.D)), 5, axis=1)
    out = O.decode_attention(rng.standard_normal((1, O.D)), hk, hv, u[None], u[None], 1)
    np.testing.assert_allclose(out[0], u @ hv[0].mean(axis=0), atol=1e-12)


# --- packed layout (library-defined) and the paper's compression figure -------------------------

@pytest.mark.parametrize("case", _gold("packing_examples.json")["cases"])
def test_pack_hand_examples(case):
    bits = np.array(case["bits"])
    codes = np.array([case["codes"]])
    words = O.pack_records(codes, bits, len(case["words"]))
    assert words[0].tolist() == case["words"]
    assert O.unpack_records(words, bits).tolist() == [case["codes"]]


@pytest.mark.parametrize("b_hi", [9, 17])
def test_pack_round_trip_random(b_hi):
    """Widths up to 8 (device plans) and up to 16 (the planner's range)."""
    rng = np.random.default_rng(14 + b_hi)
    for _ in range(20):
        bits = np.sort(rng.integers(0, b_hi, O.D))[::-1]
        half = np.where(bits > 0, 2 ** np.maximum(bits - 1, 0), 0)
        codes = np.where(bits > 0, rng.integers(-half, np.maximum(half, 1), (64, O.D)), 0)
        nw = O.record_words([bits])
        assert O.unpack_records(O.pack_records(codes, bits, nw), bits).tolist() == codes.tolist()


def test_value_interleave_round_trip():
    """Values are stored quad-interleaved in byte-quarters; keys plainly.  Writing records into a
    cache image and reading them back returns them unchanged for every token position."""
    rng = np.random.default_rng(15)
    bits = np.sort(rng.integers(1, 9, O.D))[::-1]
    nw = O.record_words([bits])
    n = 300
    codes = [rng.integers(-(2 ** (bits - 1)), 2 ** (bits - 1), (n, O.D)) for _ in range(4)]
    recs = [O.pack_records(c, bits, nw) for c in codes]
    alphas = [rng.random(n).astype(np.float32) for _ in range(4)]
    img = O.cache_image([[recs[0], recs[1]]], [[recs[2], recs[3]]], [[alphas[0], alphas[1]]],
                        [[alphas[2], alphas[3]]], 1, 2, 384, nw)
    for h in range(2):
        for kind, idx in ((0, h), (1, 2 + h)):
            rec, al = O.cache_records(img, 1, 2, 384, nw, 0, h, kind, 0, n)
            assert np.array_equal(rec, recs[idx]) and np.array_equal(al, alphas[idx])
            assert np.array_equal(O.unpack_records(rec, bits), codes[idx])
    slots = sorted(O.value_slot_of(t, r) for t in range(8) for r in range(4))
    assert slots == [(s, i) for s in range(8) for i in range(4)]


def test_value_interleave_hand_example():
    """The value layout written out by hand for one token quad: token t's record word has bytes
    16t + r (r = 0..3); slot (0, 2, 1, 3)[r] of the quad holds byte-quarter r of the four tokens,
    token i in byte i, so the slots read 0x30201000, 0x32221202, 0x31211101, 0x33231303.  Keys
    are stored plainly: slot t holds token t's word."""
    words = np.array([[sum((16 * t + r) << (8 * r) for r in range(4))] for t in range(4)], np.uint32)
    img = O.cache_image([[words]], [[words]], [[np.zeros(4, np.float32)]], [[np.zeros(4, np.float32)]],
                        1, 1, 128, 1)
    plane_k = img[0:128]
    plane_v = img[128:256]
    assert plane_v[:4].tolist() == [0x30201000, 0x32221202, 0x31211101, 0x33231303]
    assert plane_k[:4].tolist() == words[:, 0].tolist()
    assert not plane_v[4:].any() and not plane_k[4:].any()


def test_record_size_matches_paper_compression():
    g = _gold("compression_ratios.json")
    cfg = W.CONFIGS["tiny"]
    x = W.calibration_vectors(cfg, 0, 0, W.KIND_K).astype(np.float64)
    bits = O.plan_stream(x, g["avg_bits"])["bits"]
    assert int(bits.sum()) == 352                        # 2.75 * 128 code bits per token
    ratio = g["fp16_bits"] * O.D / bits.sum()
    assert round(ratio, 2) == g["ratio_printed"]
    assert g["llama_fp16_gb"] * 1000 / ratio == pytest.approx(g["llama_aatc_mb"], rel=0.005)
    assert O.record_words([bits]) == 11


def test_dequantize_f32_is_two_roundings():
    codes = np.array([[3, -2]])
    alpha = np.array([0.1], np.float32)
    s = np.array([0.3, 0.7], np.float32)
    bits = np.array([3, 2])
    got = O.dequantize_f32(codes, alpha, s, bits)
    f0 = np.float32(0.3) * np.float32(2.0 ** -2)
    f1 = np.float32(0.7) * np.float32(2.0 ** -1)
    assert got[0, 0] == np.float32(np.float32(3) * np.float32(alpha[0] * f0))
    assert got[0, 1] == np.float32(np.float32(-2) * np.float32(alpha[0] * f1))


def _rn32(x):
    """Round an exact rational to the nearest fp32 value, ties to even (normal range), with
    integer arithmetic only."""
    from fractions import Fraction
    if x == 0:
        return Fraction(0)
    sign, x = (-1 if x < 0 else 1), abs(x)
    e = x.numerator.bit_length() - x.denominator.bit_length()
    e += 1 if Fraction(2) ** (e + 1) <= x else 0
    e -= 1 if Fraction(2) ** e > x else 0
    ulp = Fraction(2) ** (e - 23)
    m = x / ulp
    fl = m.numerator // m.denominator
    rem = m - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    return sign * fl * ulp


def test_dequantize_f32_rounding_order_exact_rationals():
    """The two roundings fl32(code * fl32(alpha f_c)) checked in exact rational arithmetic, on
    inputs where one rounding of the exact product code * alpha * f_c gives a different fp32
    value (so the order of the roundings is what the case decides)."""
    from fractions import Fraction
    cases = [(1081809706, 1088184628, 8, 38), (1080294143, 1075205050, 6, 7), (1075107180, 1078175588, 8, 44)]
    for a_bits, s_bits, b, code in cases:
        alpha = np.array([a_bits], np.uint32).view(np.float32)
        scale = np.array([s_bits], np.uint32).view(np.float32)
        f = Fraction(float(scale[0])) * Fraction(2) ** (1 - b)
        two = _rn32(code * _rn32(Fraction(float(alpha[0])) * f))
        one = _rn32(code * Fraction(float(alpha[0])) * f)
        assert two != one
        got = O.dequantize_f32(np.array([[code]]), alpha, scale, np.array([b]))
        assert Fraction(float(got[0, 0])) == two


# --- prefill attention over the coded cache (Def. sdpa with a causal chunk of queries) ----------

def test_prefill_attention_equals_causal_sdpa_on_reconstructed_kv():
    """Every query row of the chunk is Def. sdpa over the reconstructed keys / values up to its own
    position: library scaled_dot_product_attention with a causal mask on K = h_K U_K^T, V = h_V U_V^T."""
    import torch
    rng = np.random.default_rng(11)
    hkv, g, n_ctx, n_q = 2, 3, 40, 12
    q0 = n_ctx - n_q
    bk = np.stack([np.linalg.qr(rng.standard_normal((O.D, O.D)))[0] for _ in range(hkv)])
    bv = np.stack([np.linalg.qr(rng.standard_normal((O.D, O.D)))[0] for _ in range(hkv)])
    hk, hv = rng.standard_normal((hkv, n_ctx, O.D)), rng.standard_normal((hkv, n_ctx, O.D))
    q = rng.standard_normal((n_q, hkv * g, O.D))
    out = O.prefill_attention(q, np.arange(q0, n_ctx), hk, hv, bk, bv, g)
    k = torch.from_numpy(np.einsum("hnc,hdc->hnd", hk, bk))
    v = torch.from_numpy(np.einsum("hnc,hdc->hnd", hv, bv))
    for j in range(hkv * g):
        h = j // g
        mask = torch.from_numpy(np.arange(n_ctx)[None, :] <= np.arange(q0, n_ctx)[:, None])
        ref = torch.nn.functional.scaled_dot_product_attention(
            torch.from_numpy(q[:, j])[None], k[h][None], v[h][None], attn_mask=mask[None]).numpy()[0]
        np.testing.assert_allclose(out[:, j], ref, rtol=1e-9, atol=1e-12)
