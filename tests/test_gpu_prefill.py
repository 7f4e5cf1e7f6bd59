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
