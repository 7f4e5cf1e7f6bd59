"""Planted mistakes in the oracle must fail a pin (no GPU).

Each case replaces one oracle function, on the CPU and for the duration of the test only, by a
variant with one plausible slip -- a dropped term or factor, a wrong sign, index or rounding, a
transposed operand, a reordered step -- and runs the pins that guard that function.  The pins
compare the oracle against what the paper and the mathematics fix (closed forms, hand examples,
brute force, library SDPA, invariants), never against the CUDA path, so a case that no pin
catches would be a hole in the oracle's pinning.
"""
import math

import numpy as np
import pytest

from oracle import aatc_oracle as O

import test_global_allocation as GA
import test_head_groups as HG
import test_oracle_pins as P
import test_sink_window as SW
import test_whitening as WH


# ---------------------------------------------------------------- the planted variants

def _second_moment_centered(x):
    x = np.asarray(x, np.float64)
    xc = x - x.mean(axis=0)
    return xc.T @ xc / x.shape[0]


def _eigenbasis_ascending(c):
    lam, vec = np.linalg.eigh(np.asarray(c, np.float64))
    return lam, O.canonical_sign(vec)


def _key_weights_abs(recon_rows, queries_by_head):
    b = np.asarray(recon_rows, np.float64)
    w = np.zeros(b.shape[0])
    for q in queries_by_head:
        w += np.mean(np.abs(np.asarray(q, np.float64) @ b.T), axis=0)
    return w


def _key_weights_transposed(recon_rows, queries_by_head):
    b = np.asarray(recon_rows, np.float64)
    w = np.zeros(b.shape[0])
    for q in queries_by_head:
        proj = np.asarray(q, np.float64) @ b
        w += np.mean(proj * proj, axis=0)
    return w


def _key_weights_head_mean(recon_rows, queries_by_head):
    qs = list(queries_by_head)
    b = np.asarray(recon_rows, np.float64)
    w = np.zeros(b.shape[0])
    for q in qs:
        proj = np.asarray(q, np.float64) @ b.T
        w += np.mean(proj * proj, axis=0)
    return w / len(qs)


def _value_weights_no_wo(recon_rows, w_o=None):
    b = np.asarray(recon_rows, np.float64)
    return np.sum(b * b, axis=1)


def _objective_base2(g, bits):
    return float(np.sum(np.asarray(g, np.float64) * np.exp2(-np.asarray(bits, np.float64))))


def _greedy_base2(g, budget, b_max):
    g = np.asarray(g, np.float64)
    bits = np.zeros(len(g), dtype=np.int64)
    for _ in range(int(budget)):
        gain = np.where(bits < b_max, g * np.exp2(-1.0 * bits), -np.inf)
        c = int(np.argmax(gain))
        if not np.isfinite(gain[c]):
            break
        bits[c] += 1
    return bits


def _greedy_no_cap(g, budget, b_max):
    g = np.asarray(g, np.float64)
    bits = np.zeros(len(g), dtype=np.int64)
    for _ in range(int(budget)):
        bits[int(np.argmax(g * np.exp2(-2.0 * bits)))] += 1
    return bits


def _continuous_no_half(g, budget, b_max=np.inf):
    g = np.asarray(g, np.float64)

    def total(lt):
        return float(np.sum(np.clip(np.log2(g) - lt, 0.0, b_max)))

    lo, hi = math.log2(g.min()) - 2 * 64, math.log2(g.max())
    for _ in range(400):
        mid = 0.5 * (lo + hi)
        if total(mid) > budget:
            lo = mid
        else:
            hi = mid
    lt = 0.5 * (lo + hi)
    return np.clip(np.log2(g) - lt, 0.0, b_max), 2.0 ** lt


def _percentile_nearest_rank(values, p):
    a = np.sort(np.asarray(values, np.float64))
    return float(a[int(round((p / 100.0) * (len(a) - 1)))])


def _scales_p95(encode_basis, x, p=95.0):
    h = np.abs(np.asarray(x, np.float64) @ encode_basis)
    return np.array([O.percentile_linear(h[:, c], p) for c in range(h.shape[1])])


def _scales_signed(encode_basis, x, p=99.0):
    h = np.asarray(x, np.float64) @ encode_basis
    return np.array([O.percentile_linear(h[:, c], p) for c in range(h.shape[1])])


def _token_scale_all_channels(h, scales, bits):
    return np.max(np.abs(h) / np.asarray(scales, np.float64), axis=1)


def _token_scale_times_s(h, scales, bits):
    keep = np.asarray(bits) > 0
    return np.max(np.abs(h[:, keep]) * np.asarray(scales, np.float64)[keep], axis=1)


def _make_quantize(rounding="half_up", clamp_hi_extra=0, delta_factor=2.0):
    def quantize(h, alpha, scales, bits):
        h = np.asarray(h, np.float64)
        b = np.asarray(bits, np.int64)
        s = np.asarray(scales, np.float64)
        keep = b > 0
        codes = np.zeros(h.shape, dtype=np.int64)
        t = np.zeros(h.shape)
        delta = delta_factor * alpha[:, None] * s[None, keep] / np.exp2(b[keep])[None, :]
        with np.errstate(divide="ignore", invalid="ignore"):
            tk = np.where(delta > 0, h[:, keep] / np.where(delta > 0, delta, 1.0), 0.0)
        if rounding == "floor":
            r = np.floor(tk)
        elif rounding == "away":
            r = np.sign(tk) * np.floor(np.abs(tk) + 0.5)
        else:
            r = np.floor(tk + 0.5)
        lo = -np.exp2(b[keep] - 1)
        hi = np.exp2(b[keep] - 1) - 1 + clamp_hi_extra
        codes[:, keep] = np.clip(r, lo, hi).astype(np.int64)
        t[:, keep] = tk
        return codes, t
    return quantize


def _dequantize_no_two(codes, alpha, scales, bits):
    b = np.asarray(bits, np.int64)
    delta = alpha[:, None] * np.asarray(scales, np.float64)[None, :] / np.exp2(b)[None, :]
    return np.where(b[None, :] > 0, codes * delta, 0.0)


def _dequantize_f32_one_rounding(codes, alpha_f32, scales_f32, bits):
    b = np.asarray(bits, np.int64)
    exact = (np.asarray(codes, np.float64) * np.asarray(alpha_f32, np.float64)[:, None] *
             np.asarray(scales_f32, np.float64)[None, :] * np.exp2(1 - b)[None, :])
    return np.where(b[None, :] > 0, exact.astype(np.float32), np.float32(0.0)).astype(np.float32)


def _record_entries_ragged(bits):
    b = [int(x) for x in bits]
    d2 = []
    for k in range(8):
        d2 += [(c, 2 * k) for c in range(len(b)) if b[c] >= 2 * k + 2]
    return d2, [(c, b[c] - 1) for c in range(len(b)) if b[c] % 2 == 1]


def _record_entries_top_bit_low(bits):
    d2, d1 = _ORIG["record_entries"](bits)
    top = {c: int(bits[c]) - 1 for c in range(len(bits)) if int(bits[c]) % 2 == 1}
    return d2, [(c, 0) if top.get(c) == sh else (c, sh) for (c, sh) in d1]


def _pack_msb_first(codes, bits, n_words):
    b = np.asarray(bits, np.int64)
    u = np.where(b[None, :] > 0, codes + np.where(b > 0, 2 ** np.maximum(b - 1, 0), 0)[None, :], 0).astype(np.uint64)
    d2, d1 = O.record_entries(b)
    words = np.zeros((codes.shape[0], n_words), dtype=np.uint64)
    for i, (c, sh) in enumerate(d2):
        words[:, i // 16] |= ((u[:, c] >> np.uint64(sh)) & np.uint64(3)) << np.uint64(30 - 2 * (i % 16))
    base = len(d2) // 16
    for j, (c, sh) in enumerate(d1):
        words[:, base + j // 32] |= ((u[:, c] >> np.uint64(sh)) & np.uint64(1)) << np.uint64(31 - j % 32)
    return words.astype(np.uint32)


def _value_slot_identity(token_in_tile, quarter):
    q, i = divmod(token_in_tile, 4)
    return 4 * q + quarter, i


def _softmax_unnormalised(s):
    s = np.asarray(s, np.float64)
    return np.exp(s - np.max(s))


def _attention_unscaled(q, k, v, w_o=None):
    q = np.asarray(q, np.float64)
    a = O.softmax(np.asarray(k, np.float64) @ q)
    o = a @ np.asarray(v, np.float64)
    return o if w_o is None else o @ np.asarray(w_o, np.float64)


def _make_decode(variant):
    def decode_attention(q_heads, hk, hv, basis_k, basis_v, group):
        out = np.zeros((q_heads.shape[0], O.D))
        for j in range(q_heads.shape[0]):
            h = j % len(hk) if variant == "head_map" else j // group     # interleaved vs blocked GQA
            bk = np.asarray(basis_k[h], np.float64)
            qt = (bk if variant == "transposed" else bk.T) @ np.asarray(q_heads[j], np.float64)
            scale = 1.0 if variant == "unscaled" else 1.0 / math.sqrt(O.D)
            a = O.softmax(np.asarray(hk[h], np.float64) @ qt * scale)
            acc = a @ np.asarray(hv[h], np.float64)
            out[j] = acc if variant == "no_value_transform" else np.asarray(basis_v[h], np.float64) @ acc
        return out
    return decode_attention


def _make_prefill(extent):
    def prefill_attention(q_tokens, positions, hk, hv, basis_k, basis_v, group):
        out = np.zeros((q_tokens.shape[0], q_tokens.shape[1], O.D))
        for i, pos in enumerate(np.asarray(positions, np.int64)):
            stop = hk.shape[1] if extent == "all" else int(pos)
            out[i] = O.decode_attention(q_tokens[i], hk[:, :stop], hv[:, :stop], basis_k, basis_v, group)
        return out
    return prefill_attention


def _make_mixed(variant):
    def decode_attention_mixed(q_heads, hk, hv, basis_k, basis_v, group, k_full, v_full):
        out = np.zeros((q_heads.shape[0], O.D))
        for j in range(q_heads.shape[0]):
            h = j // group
            q = np.asarray(q_heads[j], np.float64)
            qt = np.asarray(basis_k[h], np.float64).T @ q
            s_c = np.asarray(hk[h], np.float64) @ qt / math.sqrt(O.D)
            s_f = np.asarray(k_full[h], np.float64) @ q / (1.0 if variant == "unscaled_full" else math.sqrt(O.D))
            a = O.softmax(np.concatenate([s_c, s_f]))
            n_c = s_c.shape[0]
            full = 0.0 if variant == "no_full_values" else a[n_c:] @ np.asarray(v_full[h], np.float64)
            out[j] = np.asarray(basis_v[h], np.float64) @ (a[:n_c] @ np.asarray(hv[h], np.float64)) + full
        return out
    return decode_attention_mixed


def _sink_window_flush_at_window(n_tokens, sink=4, window=128, step=16):
    n_sink = min(n_tokens, sink)
    rest = n_tokens - n_sink
    n_coded = step * max(0, (rest - window + step) // step)
    return n_sink, n_coded, rest - n_coded


def _make_distortion(variant):
    def distortion_decomposition(q, k, v, var_k, var_v, w_o=None):
        q = np.asarray(q, np.float64)
        k = np.asarray(k, np.float64)
        v = np.asarray(v, np.float64)
        d = q.shape[-1]
        wo = np.eye(v.shape[1]) if w_o is None else np.asarray(w_o, np.float64)
        a = O.softmax(k @ q / math.sqrt(d))
        vw = v @ wo
        o = a @ vw
        qe = q if variant == "unscaled_q" else q / math.sqrt(d)
        aa = a if variant == "linear_a" else a ** 2
        resid = np.sum((vw - o) ** 2, axis=1)
        dk = float(np.sum(aa * resid * (np.asarray(var_k) @ (qe ** 2))))
        dv = float(np.sum(aa * (np.asarray(var_v) @ np.sum(wo ** 2, axis=1))))
        return dk, dv
    return distortion_decomposition


def _make_global(variant):
    def global_allocation(sigma2, weights, avg_bits_k, avg_bits_v, n_protect=3, b_max=8):
        sigma2 = np.asarray(sigma2, np.float64)
        weights = np.asarray(weights, np.float64)
        L, H, _, d = sigma2.shape
        bits = np.zeros(sigma2.shape, dtype=np.int64)
        np_ = min(n_protect, L)
        for kind, avg in ((0, avg_bits_k), (1, avg_bits_v)):
            per_stream = int(round(avg * d))
            extra = d if (kind == 0 and variant != "no_key_bonus") else 0
            prot = min(per_stream + extra, b_max * d)
            for l in range(np_):
                for h in range(H):
                    bits[l, h, kind] = O.greedy_allocation(weights[l, h, kind] * sigma2[l, h, kind], prot, b_max)
            rest = per_stream * L * H - prot * np_ * H
            if np_ == L:
                continue
            g = []
            for l in range(np_, L):
                if variant == "no_normalisation":
                    ps = pw = 1.0
                else:
                    ps = O.percentile_linear(sigma2[l, :, kind].ravel(), 95.0) or 1.0
                    pw = O.percentile_linear(weights[l, :, kind].ravel(), 95.0) or 1.0
                g.append((sigma2[l, :, kind] / ps) * (weights[l, :, kind] / pw))
            pooled = O.greedy_allocation(np.concatenate([x.ravel() for x in g]), rest, b_max)
            bits[np_:, :, kind] = pooled.reshape(L - np_, H, d)
        return bits
    return global_allocation


def _channel_variance_centered(encode_basis, x):
    h = np.asarray(x, np.float64) @ encode_basis
    return np.var(h, axis=0)


def _plan_stream_unsorted(x_calib, avg_bits, b_max=8, queries_by_head=None, weights="aatc"):
    lam, u = O.eigenbasis(O.second_moment(x_calib))
    if weights == "var":
        w = np.ones(O.D)
    elif queries_by_head is not None:
        w = O.key_weights(u.T, queries_by_head)
    else:
        w = O.value_weights(u.T)
    g = w * lam
    bits = O.greedy_allocation(g, int(round(avg_bits * O.D)), b_max)
    return {"basis": u, "bits": bits, "scales": O.channel_scales(u, x_calib), "sigma2": lam, "weights": w, "g": g}


def _embed_block0(q, block, n_blocks):
    return _ORIG["embed_query"](q, 0, n_blocks)


def _group_decode_group_scale(q_heads, hk, hv, basis_k, basis_v, group):
    hk = np.asarray(hk, np.float64)
    hv = np.asarray(hv, np.float64)
    g_h = hk.shape[1] // O.D
    out = np.zeros((q_heads.shape[0], O.D))
    for i in range(q_heads.shape[0]):
        m = i // group
        qt = np.asarray(basis_k, np.float64).T @ O.embed_query(q_heads[i], m, g_h)
        a = O.softmax(hk @ qt / math.sqrt(O.D * g_h))
        out[i] = (np.asarray(basis_v, np.float64) @ (a @ hv))[O.D * m:O.D * (m + 1)]
    return out


def _whitening_l_not_lt(x_calib, w):
    x = np.asarray(x_calib, np.float64)
    w = np.asarray(w, np.float64)
    l_chol = np.linalg.cholesky(x.T @ x / x.shape[0])
    u, s, pt = np.linalg.svd(l_chol @ w, full_matrices=False)
    p_mat = pt.T
    a = np.linalg.solve(l_chol.T, u) * np.sqrt(s)[None, :]
    return {"A": a, "B": np.sqrt(s)[:, None] * p_mat.T, "S": s, "P": p_mat, "U": u, "L": l_chol}


def _hidden_operand_times_s(a, s):
    return np.asarray(a, np.float64) * np.asarray(s, np.float64)[None, :]


# ---------------------------------------------------------------- which pins guard what

def _textbook():
    for case in P._gold("waterfill_textbook.json")["cases"]:
        P.test_continuous_waterfilling_textbook(case)


def _packing_examples():
    for case in P._gold("packing_examples.json")["cases"]:
        P.test_pack_hand_examples(case)


def _pack_round_trips():
    for b_hi in (9, 17):
        P.test_pack_round_trip_random(b_hi)


def _sink_counts():
    for args in ((4, 128, 16), (0, 32, 8), (2, 16, 16)):
        SW.test_sink_window_counts_match_token_by_token_policy(*args)


_ORIG = {}

MUTANTS = [
    # (oracle function, planted mistake, variant, pins that must catch it)
    ("second_moment", "centered covariance instead of the uncentered second moment", _second_moment_centered,
     [P.test_whitening_svd_equals_pca, HG.test_block_diagonal_second_moment_splits_into_per_head_bases]),
    ("eigenbasis", "eigenvalues ascending", _eigenbasis_ascending, [P.test_whitening_svd_equals_pca]),
    ("key_weights", "|u.q| instead of (u.q)^2", _key_weights_abs, [P.test_key_weights_gqa_hand_example]),
    ("key_weights", "transposed reconstruction basis", _key_weights_transposed, [P.test_key_weights_gqa_hand_example]),
    ("key_weights", "GQA heads averaged instead of summed", _key_weights_head_mean, [P.test_key_weights_gqa_hand_example]),
    ("value_weights", "output projection ignored", _value_weights_no_wo, [P.test_key_weights_gqa_hand_example]),
    ("allocation_objective", "2^-b instead of 4^-b", _objective_base2,
     [P.test_greedy_integer_local_optimality_and_monotone]),
    ("greedy_allocation", "marginal gain with 2^-b", _greedy_base2,
     [P.test_greedy_integer_local_optimality_and_monotone, P.test_greedy_saturates_at_b_max]),
    ("greedy_allocation", "width cap b_max ignored", _greedy_no_cap, [P.test_greedy_saturates_at_b_max]),
    ("continuous_allocation", "b = log2(g / theta), the 1/2 dropped", _continuous_no_half,
     [_textbook, P.test_continuous_waterfilling_kkt]),
    ("percentile_linear", "nearest rank instead of linear interpolation", _percentile_nearest_rank,
     [P.test_percentile_definition]),
    ("channel_scales", "95th instead of 99th percentile", _scales_p95, [P.test_channel_scale_is_p99_of_magnitudes]),
    ("channel_scales", "percentile of signed coefficients", _scales_signed, [P.test_channel_scale_is_p99_of_magnitudes]),
    ("token_scale", "maximum over dropped channels too", _token_scale_all_channels,
     [P.test_token_scale_ignores_dropped_channels]),
    ("token_scale", "h * s instead of h / s", _token_scale_times_s, [P.test_token_scale_ignores_dropped_channels]),
    ("quantize", "floor without the half", _make_quantize(rounding="floor"), [P.test_quantizer_specific_values]),
    ("quantize", "round half away from zero", _make_quantize(rounding="away"), [P.test_quantizer_specific_values]),
    ("quantize", "clamp one level too high", _make_quantize(clamp_hi_extra=1),
     [P.test_quantizer_specific_values, P.test_quantizer_error_bound_and_clamp]),
    ("quantize", "step without the factor 2", _make_quantize(delta_factor=1.0),
     [P.test_quantizer_specific_values, P.test_quantizer_error_bound_and_clamp]),
    ("dequantize", "step without the factor 2", _dequantize_no_two,
     [P.test_quantizer_error_bound_and_clamp, P.test_noise_model_high_rate]),
    ("dequantize_f32", "one rounding of the exact product", _dequantize_f32_one_rounding,
     [P.test_dequantize_f32_is_two_roundings, P.test_dequantize_f32_rounding_order_exact_rationals]),
    ("record_entries", "ragged D2 tail left in place", _record_entries_ragged,
     [_pack_round_trips, _packing_examples]),
    ("record_entries", "odd top bit taken from bit 0", _record_entries_top_bit_low,
     [_pack_round_trips, _packing_examples]),
    ("pack_records", "fields MSB-first", _pack_msb_first, [_packing_examples]),
    ("value_slot_of", "byte-quarters in slot order 0, 1, 2, 3", _value_slot_identity,
     [P.test_value_interleave_hand_example]),
    ("softmax", "no normalisation", _softmax_unnormalised, [P.test_decode_matches_library_sdpa]),
    ("attention", "scores without 1/sqrt(d)", _attention_unscaled,
     [HG.test_group_decode_with_exact_coefficients_is_plain_attention,
      SW.test_mixed_decode_is_plain_attention_when_coding_is_lossless]),
    ("decode_attention", "scores without 1/sqrt(d)", _make_decode("unscaled"), [P.test_decode_matches_library_sdpa]),
    ("decode_attention", "U_K q instead of U_K^T q", _make_decode("transposed"), [P.test_decode_matches_library_sdpa]),
    ("decode_attention", "query head j reads kv-head j mod H_kv", _make_decode("head_map"),
     [P.test_decode_matches_library_sdpa]),
    ("decode_attention", "value transform U_V dropped", _make_decode("no_value_transform"),
     [P.test_decode_matches_library_sdpa, P.test_decode_special_cases]),
    ("prefill_attention", "no causal mask", _make_prefill("all"),
     [P.test_prefill_attention_equals_causal_sdpa_on_reconstructed_kv]),
    ("prefill_attention", "a row does not see its own token", _make_prefill("exclusive"),
     [P.test_prefill_attention_equals_causal_sdpa_on_reconstructed_kv]),
    ("decode_attention_mixed", "uncompressed values dropped", _make_mixed("no_full_values"),
     [SW.test_mixed_decode_is_plain_attention_when_coding_is_lossless]),
    ("decode_attention_mixed", "uncompressed scores without 1/sqrt(d)", _make_mixed("unscaled_full"),
     [SW.test_mixed_decode_is_plain_attention_when_coding_is_lossless]),
    ("sink_window_counts", "window flushed when it reaches w, not w + step", _sink_window_flush_at_window,
     [_sink_counts]),
    ("distortion_decomposition", "a_i instead of a_i^2", _make_distortion("linear_a"),
     [P.test_theorem1_value_term_exact_for_key_free_noise]),
    ("distortion_decomposition", "key term without the 1/sqrt(d) of the score", _make_distortion("unscaled_q"),
     [P.test_theorem1_monte_carlo]),
    ("global_allocation", "no per-layer normalisation", _make_global("no_normalisation"),
     [GA.test_oracle_layer_normalisation_makes_layer_scale_irrelevant]),
    ("global_allocation", "protected key streams without the extra bit", _make_global("no_key_bonus"),
     [GA.test_oracle_protected_layers_and_budget]),
    ("channel_variance", "centered variance", _channel_variance_centered,
     [P.test_allocation_and_codes_invariant_to_column_scaling]),
    ("plan_stream", "channels left in eigenvalue order", _plan_stream_unsorted,
     [HG.test_one_head_group_is_the_per_head_plan_and_decode]),
    ("embed_query", "every query head at block 0", _embed_block0,
     [HG.test_group_decode_with_exact_coefficients_is_plain_attention]),
    ("decode_attention_head_group", "1/sqrt(128 G_h) instead of 1/sqrt(128)", _group_decode_group_scale,
     [HG.test_group_decode_with_exact_coefficients_is_plain_attention]),
    ("whitening_transform", "L instead of L^T in the whitened weight", _whitening_l_not_lt,
     [WH.test_factorization_reproduces_the_projection]),
    ("hidden_encode_operand", "columns scaled by S instead of sqrt(S)", _hidden_operand_times_s,
     [WH.test_transform_equals_the_pca_basis_of_the_hot_path]),
]


@pytest.mark.parametrize("name,mistake,variant,pins", MUTANTS,
                         ids=[f"{m[0]}:{m[1]}" for m in MUTANTS])
def test_planted_mistake_fails_a_pin(monkeypatch, name, mistake, variant, pins):
    _ORIG[name] = getattr(O, name)
    for pin in pins:                                   # every pin passes on the oracle as it is
        pin()
    monkeypatch.setattr(O, name, variant)
    caught = []
    for pin in pins:
        try:
            pin()
        except AssertionError:
            caught.append(pin.__name__)
    assert caught, f"no pin catches '{mistake}' in {name}"
