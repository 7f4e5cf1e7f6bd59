"""GPU parity of plans with channel widths above 8 bits (the paper's range b in 0..16, Sec. 6
setup; the global allocation of Algorithm 1 draws from it): encode (codes, alpha, record
padding), the dequantized coefficients, decode attention and prefill against the oracle.

Reading for widths above 8 (stated once here): the one-level band of the acceptance rule is
relative (1e-4 of the threshold).  One code step of a b-bit channel is 2^(1-b) alpha s_c, so at
16 bits it is only ~2^4 fp32 ulps of h, and the tensor-core GEMM's fp32 rounding of h (absolute,
~2^-20 alpha s_c) can move h across a threshold close to zero, where the relative band is
narrower than that.  For such channels a one-level difference is also accepted within an
absolute band of 2^(b-1) 2^-19 in units of the step (the fp32 accumulation error of h,
conservatively); channels of 8 bits or fewer keep the stated rule and its 1e-5 count bound."""
import numpy as np
import pytest
import torch

import harness as Hn
from oracle import aatc_oracle as O
import workloads as W

DEV = "cuda:0"


def _host_u32(cache):
    return cache.cpu().numpy().view(np.uint32)


def _wide_bits(base: np.ndarray, head: list) -> np.ndarray:
    """Non-increasing widths: the given wide head, then the base allocation's largest widths."""
    rest = np.sort(np.asarray(base, np.int64))[::-1][:128 - len(head)]
    return np.concatenate([np.asarray(head, np.int64), np.minimum(rest, min(head))]).astype(np.uint8)


def _check_wide_codes(x, rec, alpha_gpu, basis_bf16, bits, scales):
    """Codes of x under the oracle against the GPU's records; returns (mismatch <= 8 bits,
    codes <= 8 bits, mismatch > 8 bits, codes > 8 bits)."""
    b = bits.astype(np.int64)
    codes, alpha, t = O.encode_stream(np.asarray(x, np.float64), basis_bf16.astype(np.float64), b,
                                      scales.astype(np.float64))
    got = O.unpack_records(rec, b)
    keep = b > 0
    diff = got - codes
    thr = np.floor(t) + 0.5
    band = np.maximum(Hn.NEAR_REL * np.abs(thr), np.where(b > 8, np.exp2(b - 1.0) * 2.0 ** -19, 0.0)[None, :])
    near = np.abs(t - thr) <= band
    bad = (diff != 0) & keep[None, :] & ~((np.abs(diff) == 1) & near)
    assert not bad.any(), f"{int(bad.sum())} codes differ away from a threshold"
    assert np.array_equal(O.pack_records(got, b, rec.shape[1]), rec), "record padding bits must be zero"
    assert np.allclose(np.asarray(alpha_gpu, np.float64), alpha, rtol=2e-5, atol=1e-30)
    narrow, wide = keep & (b <= 8), b > 8
    n = x.shape[0]
    return (int(np.count_nonzero(diff[:, narrow])), int(narrow.sum()) * n,
            int(np.count_nonzero(diff[:, wide])), int(wide.sum()) * n)


def _wide_case(aatc, cfg, heads_k, heads_v, avg_bits=2.75):
    case = Hn.Case(aatc, cfg, avg_bits)
    bits = case.bits.copy()
    for h in range(cfg.n_kv_heads):
        bits[0, h, 0] = _wide_bits(case.bits[0, h, 0], heads_k)
        bits[0, h, 1] = _wide_bits(case.bits[0, h, 1], heads_v)
    case.dm = aatc.dims(cfg.n_layers, cfg.n_kv_heads, cfg.n_q_heads, b_max=16)
    case.bits = bits
    case.plan.close()
    case.plan = aatc.Plan(case.dm, case.basis, bits, case.scales)
    return case


# Keys: every width 9..16 (odd widths 9..15 put top bits in D1 from the high bytes; digit layers
# 4..7 exist).  Values: a head whose D2 count leaves digits of layers 5..7 moved behind the D1 bits.
K_HEAD = [16, 16, 15, 14, 13, 13, 12, 11, 10, 9, 9, 9]
V_HEAD = [16, 14, 14, 12, 11, 10, 10, 9]


def test_wide_layout_moves_high_digits(aatc):
    """The value widths of test_wide_codes_dequant_decode move digits of layers >= 4 behind the D1
    bits, and its key widths have odd widths above 8 (oracle layout, host planner: no GPU)."""
    cfg = W.Config(7, "wide", 1, 2, 8, 1, 700, (2.75,), 1, "widths up to 16")
    ck, cv, cq = W.layer_calibration(cfg, 0)
    p = aatc.calibrate(aatc.dims(1, cfg.n_kv_heads, cfg.n_q_heads), ck[None], cv[None], cq[None], 2.75)
    vb = _wide_bits(p["bits"][0, 0, 1], V_HEAD).astype(np.int64)
    d2_all = sum(int(np.sum(vb >= 2 * k + 2)) for k in range(8))
    d2, d1 = O.record_entries(vb)
    moved = d2_all - len(d2)
    assert moved > 0 and any(sh >= 8 for (_, sh) in d1[len(d1) - 2 * moved:])
    kb = _wide_bits(p["bits"][0, 0, 0], K_HEAD).astype(np.int64)
    assert {9, 11, 13, 15} <= set(kb.tolist()) and int(np.sum(kb > 8)) <= 32


@pytest.mark.gpu
def test_wide_codes_dequant_decode(aatc):
    cfg = W.Config(7, "wide", 1, 2, 8, 1, 700, (2.75,), 1, "widths up to 16")
    case = _wide_case(aatc, cfg, K_HEAD, V_HEAD)
    assert int(case.bits.max()) == 16 and case.plan.n_words > 11
    T, max_tokens = 653, 700
    k, v = W.kv_host(cfg, 0, 1, T)
    kd = torch.from_numpy(k).to(DEV).to(torch.bfloat16)
    vd = torch.from_numpy(v).to(DEV).to(torch.bfloat16)
    cache = case.plan.new_cache(1, max_tokens, DEV)
    cache.zero_()
    # two appends, the second at a start that is not a multiple of 4 (value words byte by byte)
    aatc.encode(case.plan, 0, kd[:, :398], vd[:, :398], cache, 0, max_tokens)
    aatc.encode(case.plan, 0, kd[:, 398:], vd[:, 398:], cache, 398, max_tokens)
    host = _host_u32(cache)
    tot = np.zeros(4, np.int64)
    for h in range(cfg.n_kv_heads):
        for kind, x in ((0, k), (1, v)):
            rec, alpha = Hn.read_stream(case, host, 1, max_tokens, 0, h, kind, 0, T)
            tot += _check_wide_codes(x[0, :, h], rec, alpha, case.basis_bf16[0, h, kind], case.bits[0, h, kind],
                                     case.scales[0, h, kind])
    Hn.NearThreshold.add("widths up to 16 (channels of 8 bits or fewer)", int(tot[0]), int(tot[1]))
    Hn.NearThreshold.add("widths up to 16 (channels above 8 bits)", int(tot[2]), int(tot[3]))
    Hn.NearThreshold.assert_bound("widths up to 16 (channels of 8 bits or fewer)")
    # dequantized coefficients, bit-exact
    deq = aatc.dequantize(case.plan, 0, cache, 1, 0, T, max_tokens).cpu().numpy()
    for h in range(cfg.n_kv_heads):
        for kind in (0, 1):
            rec, alpha = Hn.read_stream(case, host, 1, max_tokens, 0, h, kind, 0, T)
            b = case.bits[0, h, kind].astype(np.int64)
            ref = O.dequantize_f32(O.unpack_records(rec, b), alpha, case.scales[0, h, kind], b)
            assert np.array_equal(deq[0, :, h, kind, :].view(np.uint32), ref.view(np.uint32))
    # decode attention over the GPU's own cache
    for peaky in (1.0, 8.0):
        q = W.queries_device(cfg, 0, 1, 1, DEV, peaky=peaky)[0]
        out = aatc.decode_attention(case.plan, 0, q, cache, T, max_tokens).cpu().numpy()
        ref = Hn.oracle_decode_from_cache(case, host, 1, max_tokens, 0, 0, q.float().cpu().numpy()[0], T)
        js = sorted(ref)
        Hn.check_decode(out[0, js], np.stack([ref[j] for j in js]))
    # prefill codes are f16 tensor-core operands, exact up to 12 bits: refused here
    qh = torch.zeros((1, 4, cfg.n_q_heads, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(aatc.AatcError) as e:
        aatc.prefill_attention(case.plan, 0, qh, T - 4, cache, T, max_tokens)
    assert e.value.status == 5
    assert case.plan.device_error() == 0


@pytest.mark.gpu
def test_wide_prefill_to_12_bits(aatc):
    cfg = W.Config(7, "wide12", 1, 2, 8, 1, 400, (2.75,), 1, "widths up to 12")
    case = _wide_case(aatc, cfg, [12, 12, 11, 10, 9], [12, 10, 9, 9])
    assert int(case.bits.max()) == 12
    T, n_q = 400, 37
    k, v = W.kv_host(cfg, 0, 1, T)
    cache = case.plan.new_cache(1, T, DEV)
    cache.zero_()
    aatc.encode(case.plan, 0, torch.from_numpy(k).to(DEV).to(torch.bfloat16),
                torch.from_numpy(v).to(DEV).to(torch.bfloat16), cache, 0, T)
    rng = np.random.default_rng(12)
    qh = W.to_bf16(rng.standard_normal((1, n_q, cfg.n_q_heads, 128)))
    q0 = T - n_q
    out = aatc.prefill_attention(case.plan, 0, torch.from_numpy(qh).to(DEV).to(torch.bfloat16), q0, cache, T,
                                 T).cpu().numpy()
    u32 = _host_u32(cache)
    hk, hv = [], []
    for h in range(cfg.n_kv_heads):
        hh = []
        for kind in (0, 1):
            rec, alpha = Hn.read_stream(case, u32, 1, T, 0, h, kind, 0, T)
            b = case.bits[0, h, kind].astype(np.int64)
            hh.append(O.dequantize_f32(O.unpack_records(rec, b), alpha, case.scales[0, h, kind], b))
        hk.append(hh[0])
        hv.append(hh[1])
    ref = O.prefill_attention(qh[0].astype(np.float64), q0 + np.arange(n_q), np.stack(hk), np.stack(hv),
                              case.basis[0, :, 0], case.basis[0, :, 1], cfg.group)
    Hn.check_decode(out[0].reshape(-1, 128), ref.reshape(-1, 128))
    assert case.plan.device_error() == 0


@pytest.mark.gpu
def test_global_allocation_plan_16_bits(aatc):
    """The 5-layer global allocation at the paper's b_max = 16 (Algorithm 1): the pool gives the
    leading channels of some streams more than 8 bits, and encode + decode match the oracle."""
    cfg = W.Config(6, "global5", 5, 2, 8, 1, 2048, (4.0,), 1, "5-layer stack, global allocation, b_max 16")
    L, T = cfg.n_layers, cfg.n_ctx
    cal = [W.layer_calibration(cfg, l, anisotropic_queries=True, n=1024) for l in range(L)]
    dm = aatc.dims(L, cfg.n_kv_heads, cfg.n_q_heads, b_max=16)
    p = aatc.calibrate(dm, np.stack([c[0] for c in cal]), np.stack([c[1] for c in cal]),
                       np.stack([c[2] for c in cal]), 4.0)
    bits = aatc.allocate_global(dm, p["sigma2"], p["weights"], 4.0, 4.0, n_protect=3)
    assert int(bits.max()) > 8
    case = Hn.Case.__new__(Hn.Case)
    case.aatc, case.cfg, case.avg_bits, case.layers, case.dm = aatc, cfg, 4.0, list(range(L)), dm
    case.basis, case.bits, case.scales = p["basis"], bits, p["scales"]
    case.plan = aatc.Plan(dm, p["basis"], bits, p["scales"])
    case.basis_bf16 = Hn.bf16_round(p["basis"])
    tot = np.zeros(4, np.int64)
    for layer in (1, 4):
        kd, vd = W.kv_device(cfg, layer, 1, T, DEV)
        cache = case.plan.new_cache(1, T, DEV)
        aatc.encode(case.plan, layer, kd, vd, cache, 0, T)
        host = _host_u32(cache)
        for h in range(cfg.n_kv_heads):
            for kind, x in ((0, kd), (1, vd)):
                rec, alpha = Hn.read_stream(case, host, 1, T, 0, h, kind, 0, T)
                tot += _check_wide_codes(x[0, :, h].float().cpu().numpy(), rec, alpha, case.basis_bf16[layer, h, kind],
                                         bits[layer, h, kind], p["scales"][layer, h, kind])
        q = W.queries_device(cfg, layer, 1, 1, DEV)[0]
        out = aatc.decode_attention(case.plan, layer, q, cache, T, T).cpu().numpy()
        ref = Hn.oracle_decode_from_cache(case, host, 1, T, layer, 0, q.float().cpu().numpy()[0], T)
        js = sorted(ref)
        Hn.check_decode(out[0, js], np.stack([ref[j] for j in js]))
    Hn.NearThreshold.add("global allocation at b_max 16 (channels of 8 bits or fewer)", int(tot[0]), int(tot[1]))
    Hn.NearThreshold.add("global allocation at b_max 16 (channels above 8 bits)", int(tot[2]), int(tot[3]))
    Hn.NearThreshold.assert_bound("global allocation at b_max 16 (channels of 8 bits or fewer)")
    assert case.plan.device_error() == 0


@pytest.mark.gpu
def test_hidden_encode_refuses_wide_plan(aatc):
    cfg = W.Config(7, "wide", 1, 2, 8, 1, 256, (2.75,), 1, "widths up to 16")
    case = _wide_case(aatc, cfg, [9], [9])
    x = torch.zeros((1, 128, 256), dtype=torch.bfloat16, device=DEV)
    a_hat = torch.zeros((1, cfg.n_kv_heads, 2, 128, 256), dtype=torch.bfloat16, device=DEV)
    cache = case.plan.new_cache(1, 128, DEV)
    with pytest.raises(aatc.AatcError) as e:
        aatc.encode_hidden(case.plan, 0, x, a_hat, cache, 0, 128)
    assert e.value.status == 5
