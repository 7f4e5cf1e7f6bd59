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
import oracle_jobs
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
    ub = case.basis_bf16[layer, head, kind] if encode_matrix is None else encode_matrix
    st, err = oracle_jobs.code_check(x, rec, alpha_gpu, ub, bits, scales)
    assert err is None, f"{err} (layer {layer} head {head} kind {kind})"
    return st


class NearThreshold:
    """Near-threshold code counts of the full-size parity checks, per workload: codes that differ
    from the oracle by one level because their fp64 h / Delta lies within 1e-4 relative of a
    decision threshold.  conftest prints the table at the end of the run."""
    rows: dict = {}

    @classmethod
    def add(cls, name: str, mismatch: int, codes: int, near: int = 0):
        r = cls.rows.setdefault(name, [0, 0, 0])
        r[0] += mismatch
        r[1] += codes
        r[2] += near

    @classmethod
    def assert_bound(cls, name: str):
        mis, tot, _ = cls.rows[name]
        assert mis <= MAX_NEAR_FRACTION * tot, (name, mis, tot)


def layer_jobs(case: Case, layer: int, cache_path: str, batch: int, max_tokens: int, n_ctx: int, q_host, windows):
    """Specs of oracle_jobs.stream_job for every (sequence, kv-head) of one layer.
    q_host: (batch, H_q, 128) bf16-exact queries or None; windows(b, h) -> [(kind, t0, x)]."""
    cfg = case.cfg
    g = cfg.group
    specs = []
    for b in range(batch):
        for h in range(cfg.n_kv_heads):
            specs.append({
                "path": cache_path, "batch": batch, "n_kv": cfg.n_kv_heads, "max_tokens": max_tokens,
                "n_words": case.plan.n_words, "b": b, "h": h, "n_ctx": n_ctx,
                "bits": case.bits[layer, h], "scales": case.scales[layer, h], "basis": case.basis[layer, h],
                "enc": case.basis_bf16[layer, h],
                "q": None if q_host is None else q_host[b, h * g:(h + 1) * g],
                "windows": windows(b, h)})
    return specs


def collect_jobs(results, name: str, out_gpu=None, group: int = 1):
    """Raise on a code error, add the near-threshold counts to `name`, and compare the GPU's
    attention outputs out_gpu (batch, H_q, 128) with the oracle's for every query head."""
    errs = []
    for r in results:
        assert r["error"] is None, r["error"]
        for st in r["stats"]:
            NearThreshold.add(name, st["mismatch"], st["codes"], st["near"])
        if out_gpu is not None and r["out"] is not None:
            js = slice(r["h"] * group, (r["h"] + 1) * group)
            errs.append(check_decode(out_gpu[r["b"], js], r["out"]))
    return errs


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
