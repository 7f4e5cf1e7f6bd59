"""GPU parity of head-group plans (Sec. 5 Step 1, remark on multi-head attention: the g_h kv-heads
of a group share one transform over their concatenated 128 g_h channels): encode codes, alpha and
record padding of every slice slot, the dequantized slice coefficients, and decode attention
against the oracle's group attention (decode_attention_head_group) over the GPU's own cache."""
import numpy as np
import pytest
import torch

import harness as Hn
from oracle import aatc_oracle as O
import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _group_plan(aatc, cfg, g_h, avg_bits=2.75, layers=(0,)):
    """Plan every (layer, group, kind) stream (the oracle's group planner, which
    tests/test_head_groups.py pins the host planner to; it is faster at 512 channels); returns
    the device plan and the host arrays [L][n_groups][2][...]."""
    L, H, G = cfg.n_layers, cfg.n_kv_heads, cfg.group
    ng, n = H // g_h, 128 * g_h
    basis = np.zeros((L, ng, 2, n, n), np.float32)
    bits = np.zeros((L, ng, 2, n), np.uint8)
    scales = np.ones((L, ng, 2, n), np.float32)
    for l in range(L):
        if l not in layers:
            for g in range(ng):
                basis[l, g] = np.eye(n, dtype=np.float32)
                bits[l, g] = 2
            continue
        ck, cv, cq = W.layer_calibration(cfg, l, anisotropic_queries=True)
        for g in range(ng):
            hk = slice(g * g_h, (g + 1) * g_h)
            pk = O.plan_head_group(ck[hk], avg_bits, queries_by_head=list(cq[g * g_h * G:(g + 1) * g_h * G]), group=G)
            pv = O.plan_head_group(cv[hk], avg_bits, group=G)
            for kind, p in ((0, pk), (1, pv)):
                basis[l, g, kind], bits[l, g, kind], scales[l, g, kind] = p["basis"], p["bits"], p["scales"]
    dm = aatc.dims(L, H, cfg.n_q_heads)
    return aatc.GroupPlan(dm, g_h, basis, bits, scales), basis, bits, scales


def _slice_codes(u32, plan, cfg, g_h, max_tokens, b, g, kind, t0, n, bits):
    """The group stream's codes (n tokens x 128 g_h, storage order) and alpha from its slice slots."""
    codes = np.zeros((n, 128 * g_h), np.int64)
    alphas, recs = [], []
    for s in range(g_h):
        rec, alpha = O.cache_records(u32, 1, cfg.n_kv_heads, max_tokens, plan.n_words, b, g * g_h + s, kind, t0, n)
        codes[:, s::g_h] = O.unpack_records(rec, bits[s::g_h].astype(np.int64))
        alphas.append(alpha)
        recs.append(rec)
    return codes, alphas, recs


@pytest.mark.parametrize("g_h,n_kv,n_q,avg_bits", [(4, 8, 32, 2.75), (2, 4, 16, 2.75), (4, 4, 16, 5.0), (2, 2, 8, 7.0)])
def test_group_encode_decode_matches_oracle(aatc, g_h, n_kv, n_q, avg_bits):
    """2.75 bits: the common decode variant; 5 and 7 bits: more value entries per slice than one
    pair set per warp holds (the wider variant) and longer records."""
    cfg = W.Config(8, "groups", 1, n_kv, n_q, 1, 700, (avg_bits,), 1, "head-group plan")
    plan, basis, bits, scales = _group_plan(aatc, cfg, g_h, avg_bits)
    T, max_tokens = 653, 700
    k, v = W.kv_host(cfg, 0, 1, T)
    kd = torch.from_numpy(k).to(DEV).to(torch.bfloat16)
    vd = torch.from_numpy(v).to(DEV).to(torch.bfloat16)
    cache = plan.new_cache(1, max_tokens, DEV)
    cache.zero_()
    aatc.encode(plan, 0, kd[:, :398], vd[:, :398], cache, 0, max_tokens)      # two appends, the
    aatc.encode(plan, 0, kd[:, 398:], vd[:, 398:], cache, 398, max_tokens)    # second unaligned
    u32 = cache.cpu().numpy().view(np.uint32)
    ng, n = n_kv // g_h, 128 * g_h
    mis = tot = 0
    coeffs = {}
    deq = aatc.dequantize(plan, 0, cache, 1, 0, T, max_tokens).cpu().numpy()
    for g in range(ng):
        for kind, x in ((0, k), (1, v)):
            xg = x[0, :, g * g_h:(g + 1) * g_h].reshape(T, n)                  # concatenated kv-heads
            b_g = bits[0, g, kind].astype(np.int64)
            codes_ref, alpha_ref, tq = O.encode_stream(xg, Hn.bf16_round(basis[0, g, kind]).astype(np.float64), b_g,
                                                       scales[0, g, kind].astype(np.float64))
            got, alphas, recs = _slice_codes(u32, plan, cfg, g_h, max_tokens, 0, g, kind, 0, T, b_g)
            keep = b_g > 0
            diff = got - codes_ref
            thr = np.floor(tq) + 0.5
            near = np.abs(tq - thr) <= Hn.NEAR_REL * np.abs(thr)
            bad = (diff != 0) & keep[None, :] & ~((np.abs(diff) == 1) & near)
            assert not bad.any(), f"group {g} kind {kind}: {int(bad.sum())} codes differ away from a threshold"
            mis += int(np.count_nonzero(diff[:, keep]))
            tot += int(keep.sum()) * T
            for s in range(g_h):
                assert np.array_equal(alphas[s], alphas[0]), "every slice slot holds the token's alpha"
                bs = b_g[s::g_h]
                assert np.array_equal(O.pack_records(O.unpack_records(recs[s], bs), bs, recs[s].shape[1]), recs[s])
                ref = O.dequantize_f32(O.unpack_records(recs[s], bs), alphas[s], scales[0, g, kind][s::g_h], bs)
                assert np.array_equal(deq[0, :, g * g_h + s, kind, :].view(np.uint32), ref.view(np.uint32))
            assert np.allclose(alphas[0].astype(np.float64), alpha_ref, rtol=2e-5, atol=1e-30)
            h = np.zeros((T, n), np.float32)
            for s in range(g_h):
                bs = b_g[s::g_h]
                h[:, s::g_h] = O.dequantize_f32(O.unpack_records(recs[s], bs), alphas[s], scales[0, g, kind][s::g_h], bs)
            coeffs[(g, kind)] = h
    name = f"head groups (g_h {g_h}, {n_kv} kv-heads, {T} tokens, {avg_bits} bits)"
    Hn.NearThreshold.add(name, mis, tot)
    Hn.NearThreshold.assert_bound(name)
    for peaky in (1.0, 8.0):
        q = W.queries_device(cfg, 0, 1, 1, DEV, peaky=peaky)[0]
        out = aatc.decode_attention(plan, 0, q, cache, T, max_tokens).cpu().numpy()
        qh = q.float().cpu().numpy()[0]
        nq = g_h * cfg.group
        for g in range(ng):
            ref = O.decode_attention_head_group(qh[g * nq:(g + 1) * nq], coeffs[(g, 0)], coeffs[(g, 1)],
                                                basis[0, g, 0], basis[0, g, 1], cfg.group)
            Hn.check_decode(out[0, g * nq:(g + 1) * nq], ref)
    assert plan.device_error() == 0


def test_group_plan_refusals(aatc):
    cfg = W.Config(8, "groups", 1, 4, 16, 1, 256, (2.75,), 1, "head-group plan")
    plan, _, _, _ = _group_plan(aatc, cfg, 2)
    cache = plan.new_cache(1, 256, DEV)
    q = torch.zeros((1, 16, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(aatc.AatcError) as e:
        aatc.prefill_attention(plan, 0, q[:, None], 0, cache, 1, 256)
    assert e.value.status == 5
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_sw(plan, 0, q, cache, 0, 128, 256)
    assert e.value.status == 5
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention_noalloc(plan, 0, q, torch.empty((1, 16, 128), device=DEV), cache, 128, 256)
    assert e.value.status == 5


def test_group_decode_refuses_oversized_records(aatc):
    """A group plan whose slices need more value tiles per warp than the decode holds (7 bits on
    every channel of a g_h = 4 group: 3 base-4 digits and one bit per channel, 512 record entries
    per slice, 32 value tiles per warp) is refused with AATC_ERR_UNSUPPORTED before any launch;
    the output keeps its contents."""
    g_h, n_kv, n_q, T = 4, 4, 16, 256
    n = 128 * g_h
    basis = np.broadcast_to(np.eye(n, dtype=np.float32), (1, 1, 2, n, n)).copy()
    bits = np.full((1, 1, 2, n), 7, np.uint8)
    scales = np.ones((1, 1, 2, n), np.float32)
    plan = aatc.GroupPlan(aatc.dims(1, n_kv, n_q), g_h, basis, bits, scales)
    cache = plan.new_cache(1, T, DEV)
    cache.zero_()
    q = torch.zeros((1, n_q, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.full((1, n_q, 128), 3.0, dtype=torch.float32, device=DEV)
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(plan, 0, q, cache, T, T, out=out)
    assert e.value.status == 5
    torch.cuda.synchronize()
    assert bool(torch.all(out == 3.0))
    assert plan.device_error() == 0


def test_group_llama_layer_full_size(aatc):
    """The Llama-shaped layer with the paper's Llama grouping (two groups of four kv-heads, 512
    channels per group stream), 32768 tokens: every code of every slice against the oracle's
    encode of the concatenated kv-heads, and the decode of all 32 query heads."""
    cfg = W.CONFIGS["llama_layer"]
    g_h = 4
    plan, basis, bits, scales = _group_plan(aatc, cfg, g_h)
    T = cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, 1, T, DEV)
    cache = plan.new_cache(1, T, DEV)
    aatc.encode(plan, 0, kd, vd, cache, 0, T)
    u32 = cache.cpu().numpy().view(np.uint32)
    ng, n = cfg.n_kv_heads // g_h, 128 * g_h
    mis = tot = 0
    coeffs = {}
    for g in range(ng):
        for kind, x in ((0, kd), (1, vd)):
            xg = x[0, :, g * g_h:(g + 1) * g_h].float().cpu().numpy().reshape(T, n)
            b_g = bits[0, g, kind].astype(np.int64)
            codes_ref, alpha_ref, tq = O.encode_stream(xg, Hn.bf16_round(basis[0, g, kind]).astype(np.float64), b_g,
                                                       scales[0, g, kind].astype(np.float64))
            got, alphas, recs = _slice_codes(u32, plan, cfg, g_h, T, 0, g, kind, 0, T, b_g)
            keep = b_g > 0
            diff = got - codes_ref
            thr = np.floor(tq) + 0.5
            near = np.abs(tq - thr) <= Hn.NEAR_REL * np.abs(thr)
            bad = (diff != 0) & keep[None, :] & ~((np.abs(diff) == 1) & near)
            assert not bad.any(), f"group {g} kind {kind}: {int(bad.sum())} codes differ away from a threshold"
            mis += int(np.count_nonzero(diff[:, keep]))
            tot += int(keep.sum()) * T
            assert np.allclose(alphas[0].astype(np.float64), alpha_ref, rtol=2e-5, atol=1e-30)
            h = np.zeros((T, n), np.float32)
            for s in range(g_h):
                assert np.array_equal(alphas[s], alphas[0])
                bs = b_g[s::g_h]
                h[:, s::g_h] = O.dequantize_f32(O.unpack_records(recs[s], bs), alphas[s], scales[0, g, kind][s::g_h], bs)
            coeffs[(g, kind)] = h
    name = "head groups, Llama layer (2 x 4 kv-heads, 32768 tokens)"
    Hn.NearThreshold.add(name, mis, tot)
    Hn.NearThreshold.assert_bound(name)
    q = W.queries_device(cfg, 0, 1, 1, DEV)[0]
    out = aatc.decode_attention(plan, 0, q, cache, T, T).cpu().numpy()
    qh = q.float().cpu().numpy()[0]
    nq = g_h * cfg.group
    for g in range(ng):
        ref = O.decode_attention_head_group(qh[g * nq:(g + 1) * nq], coeffs[(g, 0)], coeffs[(g, 1)],
                                            basis[0, g, 0], basis[0, g, 1], cfg.group)
        Hn.check_decode(out[0, g * nq:(g + 1) * nq], ref)
    assert plan.device_error() == 0
