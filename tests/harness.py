"""Shared GPU-test plumbing: build a plan for a workload, encode, read the cache back, and
compare with the oracle under the acceptance rules.

Acceptance (stated for this method's encoding): codes bit-exact except codes whose fp64
t = h/Delta lies within 1e-4 relative of a decision threshold k + 1/2 -- those may differ by
exactly one level and must be fewer than 1e-5 of all codes; dequantized coefficients
bit-exact; attention outputs within max-abs 1e-2 and relative L2 1e-3 of the oracle's fp64
attention over the GPU's own packed cache.
"""
from __future__ import annotations

import numpy as np
import torch

from oracle import aatc_oracle as O
import workloads as W

NEAR_REL = 1e-4
MAX_NEAR_FRACTION = 1e-5
OUT_MAX_ABS = 1e-2
OUT_REL_L2 = 1e-3


def bf16_round(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(torch.float32).numpy()


class Case:
    """One calibrated layer stack of a workload with its device plan."""

    def __init__(self, aatc, cfg: W.Config, avg_bits: float, layers=None, anisotropic=False, n_calib=W.N_CALIB):
        self.aatc, self.cfg, self.avg_bits = aatc, cfg, avg_bits
        self.layers = list(range(cfg.n_layers)) if layers is None else list(layers)
        L = cfg.n_layers
        self.dm = aatc.dims(L, cfg.n_kv_heads, cfg.n_q_heads)
        basis = np.empty((L, cfg.n_kv_heads, 2, 128, 128), np.float32)
        bits = np.zeros((L, cfg.n_kv_heads, 2, 128), np.uint8)
        scales = np.ones((L, cfg.n_kv_heads, 2, 128), np.float32)
        for l in range(L):
            if l in self.layers:
                ck, cv, cq = W.layer_calibration(cfg, l, anisotropic_queries=anisotropic, n=n_calib)
                p = aatc.calibrate(aatc.dims(1, cfg.n_kv_heads, cfg.n_q_heads), ck[None], cv[None], cq[None],
                                   avg_bits)
                basis[l], bits[l], scales[l] = p["basis"][0], p["bits"][0], p["scales"][0]
            else:
                basis[l] = np.eye(128, dtype=np.float32)
                bits[l] = 2
        self.basis, self.bits, self.scales = basis, bits, scales
        self.plan = aatc.Plan(self.dm, basis, bits, scales)
        self.basis_bf16 = bf16_round(basis)

    def stream(self, layer, head, kind):
        return self.basis[layer, head, kind], self.bits[layer, head, kind], self.scales[layer, head, kind]


def read_stream(case: Case, cache_host_u32: np.ndarray, batch: int, max_tokens: int, b: int, head: int, kind: int,
                t0: int, n: int):
    rec, alpha = O.cache_records(cache_host_u32, batch, case.cfg.n_kv_heads, max_tokens, case.plan.n_words, b, head,
                                 kind, t0, n)
    return rec, alpha


def check_codes(case: Case, layer: int, head: int, kind: int, x: np.ndarray, rec: np.ndarray, alpha_gpu: np.ndarray,
                encode_matrix: np.ndarray | None = None):
    """x: (n, d_in) bf16-exact inputs of one stream; rec/alpha_gpu: the GPU's records.  The
    coefficients are h = x E with E = the plan's bf16 basis (d_in = 128), or `encode_matrix`
    (d_in x 128, e.g. the bf16 hidden-state operand).  Returns stats."""
    _, bits, scales = case.stream(layer, head, kind)
    ub = (case.basis_bf16[layer, head, kind] if encode_matrix is None else encode_matrix).astype(np.float64)
    codes, alpha, t = O.encode_stream(x.astype(np.float64), ub, bits.astype(np.int64), scales.astype(np.float64))
    got = O.unpack_records(rec, bits.astype(np.int64))
    keep = bits > 0
    diff = got[:, keep] - codes[:, keep]
    tk = t[:, keep]
    thr = np.floor(tk) + 0.5
    near = np.abs(tk - thr) <= NEAR_REL * np.abs(thr)
    bad = (diff != 0) & ~((np.abs(diff) == 1) & near)
    n_mis = int(np.count_nonzero(diff))
    assert not bad.any(), f"{int(bad.sum())} codes differ away from a threshold (layer {layer} head {head} kind {kind})"
    # stored records: bits beyond the used ones must be zero
    repacked = O.pack_records(got, bits.astype(np.int64), rec.shape[1])
    assert np.array_equal(repacked, rec), "record padding bits must be zero"
    np.testing.assert_allclose(alpha_gpu.astype(np.float64), alpha, rtol=2e-5, atol=1e-30)
    return {"codes": int(keep.sum()) * x.shape[0], "mismatch": n_mis}


def check_decode(out_gpu: np.ndarray, out_ref: np.ndarray):
    err = out_gpu.astype(np.float64) - out_ref
    max_abs = float(np.max(np.abs(err)))
    rel = float(np.linalg.norm(err) / np.linalg.norm(out_ref))
    assert max_abs <= OUT_MAX_ABS, max_abs
    assert rel <= OUT_REL_L2, rel
    return max_abs, rel


def oracle_decode_from_cache(case: Case, cache_host_u32, batch, max_tokens, layer, b, q_heads, n_ctx, heads=None):
    """Oracle attention for sequence b over the GPU's packed cache (fp32 dequant, fp64 math).
    q_heads: (H_q,128) bf16-exact.  heads: kv-heads to evaluate (default all)."""
    cfg = case.cfg
    g = cfg.group
    heads = range(cfg.n_kv_heads) if heads is None else heads
    out = {}
    for h in heads:
        hh = []
        for kind in (0, 1):
            rec, alpha = read_stream(case, cache_host_u32, batch, max_tokens, b, h, kind, 0, n_ctx)
            _, bits, scales = case.stream(layer, h, kind)
            codes = O.unpack_records(rec, bits.astype(np.int64))
            hh.append(O.dequantize_f32(codes, alpha, scales, bits.astype(np.int64)))
        qs = q_heads[h * g:(h + 1) * g]
        o = O.decode_attention(qs, hh[0][None], hh[1][None], case.basis[layer, h, 0][None],
                               case.basis[layer, h, 1][None], g)
        for i in range(g):
            out[h * g + i] = o[i]
    return out
