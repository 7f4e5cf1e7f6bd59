"""GPU parity of prefill attention over the packed cache (a causal chunk of queries; Def. sdpa
per query row) against the oracle's attention over the GPU's own dequantized codes."""
import numpy as np
import pytest
import torch

import harness as Hn
from oracle import aatc_oracle as O
import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _coeffs(case, u32, batch, max_tokens, b, n_ctx):
    hk, hv = [], []
    for h in range(case.cfg.n_kv_heads):
        hh = []
        for kind in (0, 1):
            rec, alpha = Hn.read_stream(case, u32, batch, max_tokens, b, h, kind, 0, n_ctx)
            _, bits, scales = case.stream(0, h, kind)
            hh.append(O.dequantize_f32(O.unpack_records(rec, bits.astype(np.int64)), alpha, scales,
                                       bits.astype(np.int64)))
        hk.append(hh[0])
        hv.append(hh[1])
    return np.stack(hk), np.stack(hv)


@pytest.mark.parametrize("name,batch,n_ctx,n_q", [("tiny", 1, 512, 512), ("tiny", 1, 300, 37),
                                                   ("qwen", 2, 700, 129)])
def test_prefill_matches_oracle(aatc, name, batch, n_ctx, n_q):
    cfg = W.CONFIGS[name]
    case = Hn.Case(aatc, cfg, 2.75)
    max_tokens = n_ctx + 5
    k, v = W.kv_host(cfg, 0, batch, n_ctx)
    cache = case.plan.new_cache(batch, max_tokens, DEV)
    cache.zero_()
    aatc.encode(case.plan, 0, torch.from_numpy(k).to(DEV).to(torch.bfloat16), torch.from_numpy(v).to(DEV).to(torch.bfloat16),
                cache, 0, max_tokens)
    rng = np.random.default_rng(5)
    qh = W.to_bf16(rng.standard_normal((batch, n_q, cfg.n_q_heads, 128)))
    q0 = n_ctx - n_q
    out = aatc.prefill_attention(case.plan, 0, torch.from_numpy(qh).to(DEV).to(torch.bfloat16), q0, cache, n_ctx,
                                 max_tokens).cpu().numpy()
    u32 = cache.cpu().numpy().view(np.uint32)
    g = cfg.group
    rows = np.arange(n_q) if n_q <= 40 else np.sort(np.random.default_rng(6).choice(n_q, 40, replace=False))
    for b in range(batch):
        hk, hv = _coeffs(case, u32, batch, max_tokens, b, n_ctx)
        ref = O.prefill_attention(qh[b, rows].astype(np.float64), q0 + rows, hk, hv, case.basis[0, :, 0],
                                  case.basis[0, :, 1], g)
        Hn.check_decode(out[b, rows].reshape(-1, 128), ref.reshape(-1, 128))
    assert case.plan.device_error() == 0


def test_prefill_argument_errors(aatc):
    cfg = W.CONFIGS["tiny"]
    case = Hn.Case(aatc, cfg, 2.75)
    cache = case.plan.new_cache(1, 64, DEV)
    q = torch.zeros((1, 8, cfg.n_q_heads, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(aatc.AatcError):
        aatc.prefill_attention(case.plan, 0, q, 60, cache, 64, 64)        # q_start + n_q > n_ctx
    with pytest.raises(aatc.AatcError):
        aatc.prefill_attention(case.plan, 0, q, 0, cache, 80, 64)         # n_ctx > max_tokens


def _run_prefill(aatc, case, batch, n_ctx, n_q, q_scale, seed):
    cfg = case.cfg
    max_tokens = n_ctx
    k, v = W.kv_host(cfg, 0, batch, n_ctx)
    cache = case.plan.new_cache(batch, max_tokens, DEV)
    aatc.encode(case.plan, 0, torch.from_numpy(k).to(DEV).to(torch.bfloat16), torch.from_numpy(v).to(DEV).to(torch.bfloat16),
                cache, 0, n_ctx)
    qh = W.to_bf16(q_scale * np.random.default_rng(seed).standard_normal((batch, n_q, cfg.n_q_heads, 128)))
    q0 = n_ctx - n_q
    out = aatc.prefill_attention(case.plan, 0, torch.from_numpy(qh).to(DEV).to(torch.bfloat16), q0, cache, n_ctx,
                                 max_tokens).cpu().numpy()
    return qh, q0, out, cache.cpu().numpy().view(np.uint32), max_tokens


def test_prefill_peaky_scores_rescale(aatc):
    """Queries x 24: score ranges of hundreds (log2 units), so row maxima keep jumping by more
    than the lazy-rescale threshold from tile to tile and the O rescale path runs often."""
    cfg = W.CONFIGS["qwen"]
    case = Hn.Case(aatc, cfg, 2.75)
    batch, n_ctx, n_q = 1, 1100, 300
    qh, q0, out, u32, max_tokens = _run_prefill(aatc, case, batch, n_ctx, n_q, 24.0, 11)
    rows = np.sort(np.random.default_rng(12).choice(n_q, 48, replace=False))
    hk, hv = _coeffs(case, u32, batch, max_tokens, 0, n_ctx)
    ref = O.prefill_attention(qh[0, rows].astype(np.float64), q0 + rows, hk, hv, case.basis[0, :, 0],
                              case.basis[0, :, 1], cfg.group)
    Hn.check_decode(out[0, rows].reshape(-1, 128), ref.reshape(-1, 128))
    assert case.plan.device_error() == 0


def test_prefill_qwen_full_length_sampled(aatc):
    """One sequence of the bench's prefill shape (8192 queries over 8192 cached tokens, 28 / 4
    heads): rows sampled over the whole range, including the first and the last row block."""
    cfg = W.CONFIGS["qwen"]
    case = Hn.Case(aatc, cfg, 2.75)
    batch, n_ctx = 1, cfg.n_ctx
    qh, q0, out, u32, max_tokens = _run_prefill(aatc, case, batch, n_ctx, n_ctx, 1.0, 13)
    rows = np.unique(np.concatenate([np.arange(3), n_ctx - 1 - np.arange(3),
                                     np.random.default_rng(14).choice(n_ctx, 18, replace=False)]))
    hk, hv = _coeffs(case, u32, batch, max_tokens, 0, n_ctx)
    ref = O.prefill_attention(qh[0, rows].astype(np.float64), q0 + rows, hk, hv, case.basis[0, :, 0],
                              case.basis[0, :, 1], cfg.group)
    Hn.check_decode(out[0, rows].reshape(-1, 128), ref.reshape(-1, 128))
    assert np.isfinite(out).all()
    assert case.plan.device_error() == 0


def test_prefill_second_layer_of_a_plan(aatc):
    """A two-layer plan, prefill on layer 1: the kernels index the layer's basis, scales and
    record layout (layer 0 holds a different, identity-basis plan)."""
    cfg = W.Config(7, "two_layer", 2, 2, 10, 1, 700, (2.75,), 1, "two-layer plan, prefill on layer 1")
    case = Hn.Case(aatc, cfg, 2.75, layers=[1])
    batch, n_ctx, n_q = 1, 700, 90
    k, v = W.kv_host(cfg, 1, batch, n_ctx)
    cache = case.plan.new_cache(batch, n_ctx, DEV)
    aatc.encode(case.plan, 1, torch.from_numpy(k).to(DEV).to(torch.bfloat16),
                torch.from_numpy(v).to(DEV).to(torch.bfloat16), cache, 0, n_ctx)
    qh = W.to_bf16(np.random.default_rng(21).standard_normal((batch, n_q, cfg.n_q_heads, 128)))
    q0 = n_ctx - n_q
    out = aatc.prefill_attention(case.plan, 1, torch.from_numpy(qh).to(DEV).to(torch.bfloat16), q0, cache, n_ctx,
                                 n_ctx).cpu().numpy()
    u32 = cache.cpu().numpy().view(np.uint32)
    hk, hv = [], []
    for h in range(cfg.n_kv_heads):
        hh = []
        for kind in (0, 1):
            rec, alpha = Hn.read_stream(case, u32, batch, n_ctx, 0, h, kind, 0, n_ctx)
            _, bits, scales = case.stream(1, h, kind)
            hh.append(O.dequantize_f32(O.unpack_records(rec, bits.astype(np.int64)), alpha, scales,
                                       bits.astype(np.int64)))
        hk.append(hh[0])
        hv.append(hh[1])
    rows = np.array([0, 1, 44, n_q - 2, n_q - 1])
    ref = O.prefill_attention(qh[0, rows].astype(np.float64), q0 + rows, np.stack(hk), np.stack(hv),
                              case.basis[1, :, 0], case.basis[1, :, 1], cfg.group)
    Hn.check_decode(out[0, rows].reshape(-1, 128), ref.reshape(-1, 128))
    assert case.plan.device_error() == 0
