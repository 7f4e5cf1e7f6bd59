"""aatc_decode_attention_noalloc: decode attention for callers that cannot allocate device memory
when they call (a serving runtime whose memory is all handed out up front by its own pool, or
plugin code inside a framework that hides its allocator).  It must give the same outputs as
aatc_decode_attention, call after call, while reusing the library's one fixed scratch array.

This file is named so that pytest collects it last; it builds all of its own state so that it
also passes alone in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import harness as Hn
import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda:0"


def test_noalloc_decode_matches_workspace_decode_twice(aatc):
    lib = aatc.load()
    cfg = W.CONFIGS["tiny"]
    case = Hn.Case(aatc, cfg, 2.75)
    k, v = W.kv_host(cfg, 0, 1, cfg.n_ctx)
    cache = case.plan.new_cache(1, cfg.n_ctx, DEV)
    aatc.encode(case.plan, 0, torch.from_numpy(k).to(DEV).to(torch.bfloat16),
                torch.from_numpy(v).to(DEV).to(torch.bfloat16), cache, 0, cfg.n_ctx)
    qs = W.queries_host(cfg, 0, 1, 2, peaky=4.0)
    stream = torch.cuda.current_stream().cuda_stream
    for call, n_ctx in enumerate((cfg.n_ctx, 300)):            # two calls in a row, different sizes
        q = torch.from_numpy(qs[call]).to(DEV).to(torch.bfloat16)
        ref = aatc.decode_attention(case.plan, 0, q, cache, n_ctx, cfg.n_ctx)
        out = torch.full((1, cfg.n_q_heads, 128), float("nan"), dtype=torch.float32, device=DEV)
        st = lib.aatc_decode_attention_noalloc(case.plan.handle, 0, q.data_ptr(), cache.data_ptr(), 1, n_ctx,
                                               cfg.n_ctx, out.data_ptr(), stream)
        assert st == 0, st
        torch.cuda.synchronize()
        # the same kernels with the same split plan: bit for bit the workspace decode's outputs
        assert torch.equal(out, ref), float((out - ref).abs().max())
        Hn.check_decode(out.cpu().numpy()[0], ref.cpu().numpy()[0].astype(np.float64))
    # a request whose split partials exceed the fixed scratch is refused before any launch
    need = ctypes.c_size_t()
    assert lib.aatc_decode_workspace_bytes(case.plan.handle, 64, 131072, ctypes.byref(need)) == 0
    assert need.value > 4 << 20
    assert lib.aatc_decode_attention_noalloc(case.plan.handle, 0, q.data_ptr(), cache.data_ptr(), 64, 131072,
                                             131072, out.data_ptr(), stream) == 4
