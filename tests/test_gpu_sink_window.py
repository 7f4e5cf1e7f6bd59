"""GPU parity of the sink / recent-window decode (aatc_decode_attention_sw and the
SinkWindowCache manager) against the oracle's joint softmax over coded and uncompressed tokens."""
import numpy as np
import pytest
import torch

import harness as Hn
import workloads as W
from oracle import aatc_oracle as O

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _coded(case, host, batch, max_tokens, layer, b, t0, t1):
    """Dequantized coefficients of coded tokens [t0, t1) of sequence b: (H_kv, n, 128) for K, V."""
    hk, hv = [], []
    for h in range(case.cfg.n_kv_heads):
        for kind, dst in ((0, hk), (1, hv)):
            rec, alpha = Hn.read_stream(case, host, batch, max_tokens, b, h, kind, t0, t1 - t0)
            _, bits, scales = case.stream(layer, h, kind)
            codes = O.unpack_records(rec, bits.astype(np.int64))
            dst.append(O.dequantize_f32(codes, alpha, scales, bits.astype(np.int64)))
    return np.stack(hk), np.stack(hv)


def _oracle(case, host, batch, max_tokens, layer, b, q, t0, t1, kf, vf):
    """kf, vf: (n_full, H_kv, 128) float arrays of the uncompressed tokens of sequence b."""
    hk, hv = _coded(case, host, batch, max_tokens, layer, b, t0, t1)
    return O.decode_attention_mixed(q, hk, hv, case.basis[layer, :, 0], case.basis[layer, :, 1], case.cfg.group,
                                    np.transpose(kf, (1, 0, 2)), np.transpose(vf, (1, 0, 2)))


@pytest.mark.parametrize("t_first,t_end,n_full", [(4, 382, 134), (4, 512, 4), (0, 300, 0), (130, 130, 70),
                                                  (127, 129, 5)])
def test_sw_decode_matches_oracle(aatc, t_first, t_end, n_full):
    cfg = W.CONFIGS["tiny"]
    case = Hn.Case(aatc, cfg, 2.75)
    T = cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, 1, T, DEV)
    cache = case.plan.new_cache(1, T, DEV)
    aatc.encode(case.plan, 0, kd, vd, cache, 0, T)
    host = cache.cpu().numpy().view(np.uint32)
    # uncompressed tokens: the first 4 and the last n_full - 4 of the sequence (any order works),
    # stored in a buffer with spare capacity
    idx = list(range(min(4, n_full))) + list(range(T - (n_full - min(4, n_full)), T))
    cap = n_full + 7
    kf = torch.zeros((1, cap, cfg.n_kv_heads, 128), dtype=torch.bfloat16, device=DEV)
    vf = torch.zeros_like(kf)
    if n_full:
        kf[:, :n_full] = kd[:, idx]
        vf[:, :n_full] = vd[:, idx]
    q = W.queries_device(cfg, 0, 1, 1, DEV, peaky=4.0)[0]
    out = aatc.decode_attention_sw(case.plan, 0, q, cache, t_first, t_end, T, kf if n_full else None,
                                   vf if n_full else None, n_full).cpu().numpy()
    ref = _oracle(case, host, 1, T, 0, 0, q.float().cpu().numpy()[0], t_first, t_end,
                  kf[0, :n_full].float().cpu().numpy(), vf[0, :n_full].float().cpu().numpy())
    Hn.check_decode(out[0], ref)


def test_sw_decode_rejects_bad_ranges(aatc):
    cfg = W.CONFIGS["tiny"]
    case = Hn.Case(aatc, cfg, 2.75)
    cache = case.plan.new_cache(1, cfg.n_ctx, DEV)
    q = W.queries_device(cfg, 0, 1, 1, DEV)[0]
    with pytest.raises(RuntimeError):
        aatc.decode_attention_sw(case.plan, 0, q, cache, 10, 5, cfg.n_ctx)            # t_first > t_end
    with pytest.raises(RuntimeError):
        aatc.decode_attention_sw(case.plan, 0, q, cache, 7, 7, cfg.n_ctx)             # nothing to attend
    with pytest.raises(RuntimeError):
        aatc.decode_attention_sw(case.plan, 0, q, cache, 0, cfg.n_ctx + 1, cfg.n_ctx)  # past capacity


def test_sink_window_cache_streaming(aatc):
    """Prefill 2000 tokens, then append in pieces of 1..40 tokens with a decode after each: the
    manager's coded range, sink and window give the oracle's joint softmax at every step."""
    from paper_2608_14191_gb300.sink_window import SinkWindowCache
    cfg = W.Config(7, "sw_stream", 1, 2, 8, 2, 2600, (2.75,), 1, "sink/window streaming")
    case = Hn.Case(aatc, cfg, 2.75, n_calib=1024)
    B, T = cfg.batch, cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, B, T, DEV)
    qs = W.queries_device(cfg, 0, B, 8, DEV, peaky=3.0)
    swc = SinkWindowCache(case.plan, 0, B, T, DEV)
    pieces = [2000] + [1, 1, 16, 15, 40, 7, 1] * 3
    n = 0
    for step, m in enumerate(pieces):
        swc.append(kd[:, n:n + m], vd[:, n:n + m])
        n += m
        if step % 4 != 0 and step != len(pieces) - 1:
            continue
        st = swc.state
        assert (st.n_sink, st.n_coded, st.n_window) == O.sink_window_counts(n)
        q = qs[step % 8]
        out = swc.decode(q).cpu().numpy()
        host = swc.cache.cpu().numpy().view(np.uint32)
        for b in range(B):
            full_idx = list(range(st.n_sink)) + list(range(st.sink + st.n_coded, n))
            ref = _oracle(case, host, B, T, 0, b, q.float().cpu().numpy()[b], st.sink, st.sink + st.n_coded,
                          kd[b, full_idx].float().cpu().numpy(), vd[b, full_idx].float().cpu().numpy())
            Hn.check_decode(out[b], ref)
    assert case.plan.device_error() == 0


def test_sw_decode_llama_layer_full_size(aatc):
    """Llama-shaped layer at 32768 tokens with the paper's policy: sink 4, window 140, coded
    [4, 32628); every kv-head and query head against the oracle."""
    cfg = W.CONFIGS["llama_layer"]
    case = Hn.Case(aatc, cfg, 2.75)
    T = cfg.n_ctx
    n_sink, n_coded, n_win = O.sink_window_counts(T)
    kd, vd = W.kv_device(cfg, 0, 1, T, DEV)
    cache = case.plan.new_cache(1, T, DEV)
    aatc.encode(case.plan, 0, kd[:, n_sink:n_sink + n_coded].contiguous(), vd[:, n_sink:n_sink + n_coded].contiguous(),
                cache, n_sink, T)
    host = cache.cpu().numpy().view(np.uint32)
    full_idx = list(range(n_sink)) + list(range(n_sink + n_coded, T))
    kf = kd[:, full_idx].contiguous()
    vf = vd[:, full_idx].contiguous()
    q = W.queries_device(cfg, 0, 1, 1, DEV)[0]
    out = aatc.decode_attention_sw(case.plan, 0, q, cache, n_sink, n_sink + n_coded, T, kf, vf,
                                   len(full_idx)).cpu().numpy()
    qh = q.float().cpu().numpy()[0]
    for h in range(cfg.n_kv_heads):
        rk, ak = Hn.read_stream(case, host, 1, T, 0, h, 0, n_sink, n_coded)
        rv, av = Hn.read_stream(case, host, 1, T, 0, h, 1, n_sink, n_coded)
        _, bk, sk = case.stream(0, h, 0)
        _, bv, sv_ = case.stream(0, h, 1)
        hk = O.dequantize_f32(O.unpack_records(rk, bk.astype(np.int64)), ak, sk, bk.astype(np.int64))
        hv = O.dequantize_f32(O.unpack_records(rv, bv.astype(np.int64)), av, sv_, bv.astype(np.int64))
        G = cfg.group
        js = list(range(h * G, (h + 1) * G))
        ref = O.decode_attention_mixed(qh[js], hk[None], hv[None],
                                       case.basis[0, h:h + 1, 0], case.basis[0, h:h + 1, 1], G,
                                       np.transpose(kf[0, :, h:h + 1].float().cpu().numpy(), (1, 0, 2)),
                                       np.transpose(vf[0, :, h:h + 1].float().cpu().numpy(), (1, 0, 2)))
        Hn.check_decode(out[0, js], ref)
    assert case.plan.device_error() == 0
