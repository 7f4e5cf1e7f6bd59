"""GPU parity of the CUDA path (through the C ABI) against the fp64 oracle.

Small cases are compared element by element; the full-size workloads are compared on every
kv-head, sequence, layer and query head, in the launch configuration the bench uses.
"""
import os
import tempfile

import numpy as np
import pytest
import torch

import harness as Hn
import oracle_jobs
from oracle import aatc_oracle as O
import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def _host_u32(cache):
    torch.cuda.synchronize()
    return cache.cpu().numpy().view(np.uint32)


def _encode_host_kv(aatc, case, k, v, batch, max_tokens, start=0, cache=None, layer=0):
    if cache is None:
        cache = case.plan.new_cache(batch, max_tokens, DEV)
        cache.zero_()
    kd = torch.from_numpy(k).to(DEV).to(torch.bfloat16).contiguous()
    vd = torch.from_numpy(v).to(DEV).to(torch.bfloat16).contiguous()
    aatc.encode(case.plan, layer, kd, vd, cache, start, max_tokens)
    return cache


# ----------------------------------------------------------------------------- tiny, element-wise

@pytest.fixture(scope="module")
def tiny(aatc):
    cfg = W.CONFIGS["tiny"]
    case = Hn.Case(aatc, cfg, 2.75)
    k, v = W.kv_host(cfg, 0, cfg.batch, cfg.n_ctx)
    cache = _encode_host_kv(aatc, case, k, v, cfg.batch, cfg.n_ctx)
    return case, k, v, cache


def test_tiny_codes_alpha_and_dequant(aatc, tiny):
    case, k, v, cache = tiny
    cfg = case.cfg
    host = _host_u32(cache)
    stats = []
    for kind, x in ((0, k), (1, v)):
        rec, alpha = Hn.read_stream(case, host, 1, cfg.n_ctx, 0, 0, kind, 0, cfg.n_ctx)
        stats.append(Hn.check_codes(case, 0, 0, kind, x[0, :, 0, :], rec, alpha))
    for st in stats:
        Hn.NearThreshold.add("tiny (512 tokens, 1 kv-head)", st["mismatch"], st["codes"], st["near"])
    Hn.NearThreshold.assert_bound("tiny (512 tokens, 1 kv-head)")
    # dequantized coefficients, bit-exact
    deq = aatc.dequantize(case.plan, 0, cache, 1, 0, cfg.n_ctx, cfg.n_ctx).cpu().numpy()
    for kind in (0, 1):
        rec, alpha = Hn.read_stream(case, host, 1, cfg.n_ctx, 0, 0, kind, 0, cfg.n_ctx)
        _, bits, scales = case.stream(0, 0, kind)
        ref = O.dequantize_f32(O.unpack_records(rec, bits.astype(np.int64)), alpha, scales, bits.astype(np.int64))
        assert np.array_equal(deq[0, :, 0, kind, :].view(np.uint32), ref.view(np.uint32))
    assert case.plan.device_error() == 0


@pytest.mark.parametrize("peaky", [1.0, 8.0])
def test_tiny_decode(aatc, tiny, peaky):
    case, k, v, cache = tiny
    cfg = case.cfg
    host = _host_u32(cache)
    qs = W.queries_host(cfg, 0, cfg.batch, 3, peaky=peaky)
    for step in range(3):
        q = torch.from_numpy(qs[step]).to(DEV).to(torch.bfloat16)
        for n_ctx in (cfg.n_ctx, 1, 200):
            out = aatc.decode_attention(case.plan, 0, q, cache, n_ctx, cfg.n_ctx).cpu().numpy()
            ref = Hn.oracle_decode_from_cache(case, host, 1, cfg.n_ctx, 0, 0, qs[step, 0], n_ctx)
            Hn.check_decode(out[0], np.stack([ref[j] for j in range(cfg.n_q_heads)]))


def test_tiny_bf16_reference_decode(aatc, tiny):
    case, k, v, cache = tiny
    cfg = case.cfg
    qs = W.queries_host(cfg, 0, 1, 1, peaky=4.0)
    kd = torch.from_numpy(k).to(DEV).to(torch.bfloat16)
    vd = torch.from_numpy(v).to(DEV).to(torch.bfloat16)
    for n_ctx in (512, 129, 1):
        out = aatc.bf16_decode_attention(kd, vd, torch.from_numpy(qs[0]).to(DEV).to(torch.bfloat16), n_ctx)
        out = out.cpu().numpy()[0]
        for j in range(cfg.n_q_heads):
            ref = O.attention(qs[0, 0, j], k[0, :n_ctx, 0], v[0, :n_ctx, 0])
            np.testing.assert_allclose(out[j], ref, atol=2e-5, rtol=1e-4)


def test_bf16_reference_decode_qwen_group7(aatc):
    """The uncompressed reference decode with G = 7 (query columns padded to 8, its own split
    plan), two sequences, a ragged context, against plain attention per query head."""
    cfg = W.CONFIGS["qwen"]
    batch, n_ctx = 2, 3000
    k, v = W.kv_host(cfg, 0, batch, n_ctx)
    qs = W.queries_host(cfg, 0, batch, 1)[0]                     # (batch, H_q, 128)
    kd = torch.from_numpy(k).to(DEV).to(torch.bfloat16)
    vd = torch.from_numpy(v).to(DEV).to(torch.bfloat16)
    out = aatc.bf16_decode_attention(kd, vd, torch.from_numpy(qs).to(DEV).to(torch.bfloat16), n_ctx - 17)
    out = out.cpu().numpy()
    g = cfg.group
    for b in range(batch):
        for j in range(0, cfg.n_q_heads, 3):
            ref = O.attention(qs[b, j], k[b, :n_ctx - 17, j // g], v[b, :n_ctx - 17, j // g])
            np.testing.assert_allclose(out[b, j], ref, atol=2e-5, rtol=1e-4)


def test_append_in_pieces_equals_one_shot(aatc, tiny):
    """Position-addressed layout: appending 300 + 1 + 211 tokens (ragged, crossing tile
    boundaries) writes the same bytes as one encode of 512 (Alg. 1 'Append')."""
    case, k, v, cache = tiny
    max_tokens = 512
    c2 = case.plan.new_cache(1, max_tokens, DEV)
    c2.fill_(-1)
    for s, e in ((0, 300), (300, 301), (301, 512)):
        _encode_host_kv(aatc, case, k[:, s:e], v[:, s:e], 1, max_tokens, start=s, cache=c2)
    assert torch.equal(c2, cache)


def test_nonfinite_input_sets_device_flag(aatc, tiny):
    case, k, v, _ = tiny
    kk = k[:, :4].copy()
    kk[0, 2, 0, 5] = np.inf
    cache = case.plan.new_cache(1, 128, DEV)
    _encode_host_kv(aatc, case, kk, v[:, :4], 1, 128, cache=cache)
    assert case.plan.device_error(clear=True) & 1
    assert case.plan.device_error() == 0


def test_bounded_wait_times_out_with_error_status(aatc, tiny):
    """A wait on an mbarrier that nothing arrives on gives up after its limit (here 2 ms), sets bit
    1 of the device flags and returns; the context stays usable (a decode afterwards still
    matches the one before)."""
    case, k, v, cache = tiny
    q = torch.from_numpy(W.to_bf16(np.random.default_rng(3).standard_normal((1, case.cfg.n_q_heads, 128)))).to(DEV).to(torch.bfloat16)
    before = aatc.decode_attention(case.plan, 0, q, cache, case.cfg.n_ctx, case.cfg.n_ctx).clone()
    flags = torch.zeros(1, dtype=torch.int32, device=DEV)
    s = torch.cuda.current_stream()
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(s)
    aatc.selftest_bounded_wait(2000, flags, s)
    t1.record(s)
    torch.cuda.synchronize()
    assert int(flags.item()) == 2
    assert 1.9 <= t0.elapsed_time(t1) < 500.0
    after = aatc.decode_attention(case.plan, 0, q, cache, case.cfg.n_ctx, case.cfg.n_ctx)
    torch.cuda.synchronize()
    assert torch.equal(before, after)
    assert case.plan.device_error() == 0
    with pytest.raises(aatc.AatcError):
        aatc.selftest_bounded_wait(0, flags, s)


def test_argument_errors_leave_outputs_untouched(aatc, tiny):
    case, k, v, cache = tiny
    q = torch.zeros((1, 4, 128), dtype=torch.bfloat16, device=DEV)
    out = torch.full((1, 4, 128), 7.0, device=DEV)
    ws = torch.empty(4, dtype=torch.float32, device=DEV)        # too small
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(case.plan, 0, q, cache, 512, 512, out=out, workspace=ws)
    assert e.value.status == 4
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(case.plan, 0, q, cache, 513, 512, out=out)
    assert e.value.status == 3
    with pytest.raises(aatc.AatcError) as e:
        aatc.decode_attention(case.plan, 1, q, cache, 10, 512, out=out)
    assert e.value.status == 1
    kd = torch.zeros((1, 10, 1, 128), dtype=torch.bfloat16, device=DEV)
    with pytest.raises(aatc.AatcError) as e:
        aatc.encode(case.plan, 0, kd, kd, cache, 505, 512)
    assert e.value.status == 3
    with pytest.raises(aatc.AatcError) as e:                   # empty context: no softmax to take
        aatc.decode_attention(case.plan, 0, q, cache, 0, 512, out=out, workspace=torch.empty(1 << 20, device=DEV))
    assert e.value.status == 1
    assert torch.all(out == 7.0)
    # an empty append (the data pointer of an empty tensor is NULL) is a no-op at any position
    before = cache.clone()
    empty = torch.empty((1, 0, 1, 128), dtype=torch.bfloat16, device=DEV)
    for start in (0, 300, 512):
        aatc.encode(case.plan, 0, empty, empty, cache, start, 512)
    torch.cuda.synchronize()
    assert torch.equal(cache, before)


# ----------------------------------------------------------------------------- full-size workloads
#
# Every kv-head of every sequence (and every layer of the stack) is compared with the oracle in
# the launch configuration the bench times: codes and alpha over the whole context (a head and
# tail window per stream on the 32-layer stack), and the attention outputs of every query head.
# The oracle side runs in spawned worker processes (tests/oracle_jobs.py) over a file image of
# the GPU's packed cache.

def _save_image(cache, td, name):
    path = os.path.join(td, name + ".npy")
    np.save(path, _host_u32(cache))
    return path


def _full_case_check(aatc, pool, cfg, avg_bits, name, decode_steps=2):
    case = Hn.Case(aatc, cfg, avg_bits)
    B, T = cfg.batch, cfg.n_ctx
    kd, vd = W.kv_device(cfg, 0, B, T, DEV)
    cache = case.plan.new_cache(B, T, DEV)
    aatc.encode(case.plan, 0, kd, vd, cache, 0, T)
    qs = W.queries_device(cfg, 0, B, decode_steps, DEV)
    outs = [aatc.decode_attention(case.plan, 0, qs[s], cache, T, T).cpu().numpy() for s in range(decode_steps)]
    kh, vh = kd.float().cpu().numpy(), vd.float().cpu().numpy()
    errs = []
    with tempfile.TemporaryDirectory() as td:
        path = _save_image(cache, td, "layer0")
        for s in range(decode_steps):
            def windows(b, h, s=s):
                return [(0, 0, kh[b, :, h]), (1, 0, vh[b, :, h])] if s == 0 else []
            specs = Hn.layer_jobs(case, 0, path, B, T, T, qs[s].float().cpu().numpy(), windows)
            errs += Hn.collect_jobs(pool.map(oracle_jobs.stream_job, specs), name, outs[s], cfg.group)
    assert len(errs) == decode_steps * B * cfg.n_kv_heads
    Hn.NearThreshold.assert_bound(name)
    assert case.plan.device_error() == 0
    return case, kd, vd, cache, errs


def test_llama_layer_full_size(aatc, oracle_pool):
    case, kd, vd, cache, _ = _full_case_check(aatc, oracle_pool, W.CONFIGS["llama_layer"], 2.75,
                                              "llama layer (32768 x 8 kv-heads, 2.75 bits)")
    # repeated calls are bitwise identical: fixed split ranges, fixed merge order, and no shared
    # state between calls beyond the workspace (a race between phases would show up here)
    cfg = W.CONFIGS["llama_layer"]
    q = W.queries_device(cfg, 0, cfg.batch, 1, DEV)[0]
    ws = torch.empty(case.plan.workspace_bytes(cfg.batch, cfg.n_ctx) // 4 + 1, dtype=torch.float32, device=DEV)
    first = aatc.decode_attention(case.plan, 0, q, cache, cfg.n_ctx, cfg.n_ctx, workspace=ws).cpu()
    for _ in range(6):
        again = aatc.decode_attention(case.plan, 0, q, cache, cfg.n_ctx, cfg.n_ctx, workspace=ws).cpu()
        assert torch.equal(first, again)


def test_qwen_batched_full_size(aatc, oracle_pool):
    _full_case_check(aatc, oracle_pool, W.CONFIGS["qwen"], 2.75, "qwen layer (16 x 8192 x 4 kv-heads, G = 7)",
                     decode_steps=1)


@pytest.mark.parametrize("avg_bits", [1.5, 2.0, 2.75, 4.0])
def test_sweep_full_size(aatc, oracle_pool, avg_bits):
    cfg = W.CONFIGS["sweep"]
    case, kd, vd, cache, _ = _full_case_check(aatc, oracle_pool, cfg, avg_bits,
                                              f"sweep (4 x 32768 x 8 kv-heads) at {avg_bits} bits", decode_steps=1)
    if avg_bits == 1.5:
        assert (case.plan.retained < 128).any()        # zero-bit channels are dropped
    # own bf16 reference decode on the same shape, every sequence and query head
    q = W.queries_device(cfg, 0, cfg.batch, 1, DEV)[0]
    out = aatc.bf16_decode_attention(kd, vd, q, cfg.n_ctx).cpu().numpy()
    qh = q.float().cpu().numpy()
    kh, vh = kd.float().cpu().numpy(), vd.float().cpu().numpy()
    for b in range(cfg.batch):
        for j in range(cfg.n_q_heads):
            h = j // cfg.group
            ref = O.attention(qh[b, j], kh[b, :, h], vh[b, :, h])
            np.testing.assert_allclose(out[b, j], ref, atol=1e-4, rtol=1e-3)


def test_llama_stack_full_size(aatc, oracle_pool):
    """32 layers x 131072 tokens, a separately calibrated plan per layer: encode layer by layer,
    then one decode step through all layers.  Every layer, kv-head and query head is compared
    with the oracle: codes and alpha on the first 512 and the last 2048 tokens of every stream,
    attention over the whole context."""
    cfg = W.CONFIGS["llama_stack"]
    name = "llama stack (32 layers x 131072 x 8 kv-heads)"
    case = Hn.Case(aatc, cfg, 2.75, layers=range(cfg.n_layers))
    T = cfg.n_ctx
    q = W.queries_device(cfg, 0, 1, 1, DEV)[0]
    qh = q.float().cpu().numpy()
    pending = []
    errs = []
    with tempfile.TemporaryDirectory() as td:
        for l in range(cfg.n_layers):
            kd, vd = W.kv_device(cfg, l, 1, T, DEV)
            cache = case.plan.new_cache(1, T, DEV)
            aatc.encode(case.plan, l, kd, vd, cache, 0, T)
            out = aatc.decode_attention(case.plan, l, q, cache, T, T).cpu().numpy()
            heads = {}
            for kind, x in ((0, kd), (1, vd)):
                heads[kind] = (x[0, :512].float().cpu().numpy(), x[0, T - 2048:].float().cpu().numpy())

            def windows(b, h, heads=heads):
                return [(kind, t0, heads[kind][i][:, h]) for kind in (0, 1)
                        for i, t0 in ((0, 0), (1, T - 2048))]
            path = _save_image(cache, td, f"layer{l}")
            del kd, vd, cache
            specs = Hn.layer_jobs(case, l, path, 1, T, T, qh, windows)
            pending.append((path, out, pool_map_async(oracle_pool, specs)))
            while len(pending) > 3:                   # bound the images held on disk
                path0, out0, r = pending.pop(0)
                errs += Hn.collect_jobs(r.get(), name, out0, cfg.group)
                os.unlink(path0)
        for path0, out0, r in pending:
            errs += Hn.collect_jobs(r.get(), name, out0, cfg.group)
    assert len(errs) == cfg.n_layers * cfg.n_kv_heads
    Hn.NearThreshold.assert_bound(name)
    assert case.plan.device_error() == 0


def pool_map_async(pool, specs):
    return pool.map_async(oracle_jobs.stream_job, specs)


def test_global_allocation_plan(aatc):
    """A 5-layer stack planned with the global cross-layer allocation (protected first 3 layers,
    one pool for the rest): streams get unequal bit totals, every record is padded to the
    plan-wide W, and encode + decode still match the oracle on a protected and a pooled layer."""
    cfg = W.Config(6, "global5", 5, 2, 8, 1, 2048, (2.75,), 1, "5-layer stack, global allocation")
    L, T = cfg.n_layers, cfg.n_ctx
    cal = [W.layer_calibration(cfg, l, anisotropic_queries=True, n=1024) for l in range(L)]
    dm = aatc.dims(L, cfg.n_kv_heads, cfg.n_q_heads)
    p = aatc.calibrate(dm, np.stack([c[0] for c in cal]), np.stack([c[1] for c in cal]),
                       np.stack([c[2] for c in cal]), 2.75)
    bits = aatc.allocate_global(dm, p["sigma2"], p["weights"], 2.75, 2.75, n_protect=3)
    per_stream = bits.astype(np.int64).sum(axis=-1)
    assert per_stream[:, :, 1].sum() == 352 * L * cfg.n_kv_heads
    assert len(np.unique(per_stream[3:])) > 1                      # the pool spreads bits unevenly
    case = Hn.Case.__new__(Hn.Case)
    case.aatc, case.cfg, case.avg_bits, case.layers, case.dm = aatc, cfg, 2.75, list(range(L)), dm
    case.basis, case.bits, case.scales = p["basis"], bits, p["scales"]
    case.plan = aatc.Plan(dm, p["basis"], bits, p["scales"])
    case.basis_bf16 = Hn.bf16_round(p["basis"])
    for layer in (1, 4):
        kd, vd = W.kv_device(cfg, layer, 1, T, DEV)
        cache = case.plan.new_cache(1, T, DEV)
        aatc.encode(case.plan, layer, kd, vd, cache, 0, T)
        host = _host_u32(cache)
        for h in range(cfg.n_kv_heads):
            for kind, x in ((0, kd), (1, vd)):
                rec, alpha = Hn.read_stream(case, host, 1, T, 0, h, kind, T - 512, 512)
                st = Hn.check_codes(case, layer, h, kind, x[0, T - 512:, h].float().cpu().numpy(), rec, alpha)
                Hn.NearThreshold.add("global allocation (5 layers, 2 kv-heads)", st["mismatch"], st["codes"],
                                     st["near"])
        q = W.queries_device(cfg, layer, 1, 1, DEV)[0]
        out = aatc.decode_attention(case.plan, layer, q, cache, T, T).cpu().numpy()
        ref = Hn.oracle_decode_from_cache(case, host, 1, T, layer, 0, q.float().cpu().numpy()[0], T)
        js = sorted(ref)
        Hn.check_decode(out[0, js], np.stack([ref[j] for j in js]))
    Hn.NearThreshold.assert_bound("global allocation (5 layers, 2 kv-heads)")
    assert case.plan.device_error() == 0
