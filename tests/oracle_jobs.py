"""Per-stream oracle checks that run in worker processes (numpy only, no torch, no CUDA).

The full-size parity tests hand every (sequence, kv-head) of a layer to a pool of spawned
workers: each worker reads the GPU's packed cache image from a file, re-encodes its share of
the input with the oracle (codes and alpha), and computes the oracle's fp64 attention over the
GPU's own packed cache for the query heads of its group.  The acceptance rules are the ones of
``harness``: codes bit-exact except one-level differences within 1e-4 relative of a decision
threshold, record padding zero, alpha to fp32 rounding; attention checked by the caller.
"""
from __future__ import annotations

import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from oracle import aatc_oracle as O  # noqa: E402

NEAR_REL = 1e-4


def code_check(x, rec, alpha_gpu, encode_matrix, bits, scales):
    """Codes of x (n, d_in) under the oracle against the GPU's records (n, W) and alpha (n,).
    Returns (stats dict, error string or None)."""
    bits = np.asarray(bits).astype(np.int64)
    codes, alpha, t = O.encode_stream(np.asarray(x, np.float64), np.asarray(encode_matrix, np.float64), bits,
                                      np.asarray(scales, np.float64))
    got = O.unpack_records(rec, bits)
    keep = bits > 0
    diff = got[:, keep] - codes[:, keep]
    tk = t[:, keep]
    thr = np.floor(tk) + 0.5
    near = np.abs(tk - thr) <= NEAR_REL * np.abs(thr)
    bad = (diff != 0) & ~((np.abs(diff) == 1) & near)
    stats = {"codes": int(keep.sum()) * x.shape[0], "mismatch": int(np.count_nonzero(diff)),
             "near": int(np.count_nonzero(near))}
    if bad.any():
        return stats, f"{int(bad.sum())} codes differ away from a threshold"
    if not np.array_equal(O.pack_records(got, bits, rec.shape[1]), rec):
        return stats, "record padding bits must be zero"
    a_gpu = np.asarray(alpha_gpu, np.float64)
    if not np.allclose(a_gpu, alpha, rtol=2e-5, atol=1e-30):
        return stats, f"alpha differs: max rel {float(np.max(np.abs(a_gpu - alpha) / np.maximum(alpha, 1e-30))):.3e}"
    return stats, None


def stream_job(spec: dict) -> dict:
    """One (layer, sequence b, kv-head h) of a packed cache image on disk.

    spec: path (cache image .npy, uint32), batch, n_kv, max_tokens, n_words, b, h, n_ctx,
          bits (2, 128), scales (2, 128), basis (2, 128, 128) fp32, enc (2, 128, 128) encode
          matrices, q (G, 128) or None, windows: list of (kind, t0, x (n, 128)).
    Returns dict(b, h, out (G, 128) or None, stats {kind: ...}, error)."""
    img = np.load(spec["path"], mmap_mode="r")
    res = {"b": spec["b"], "h": spec["h"], "out": None, "stats": [], "error": None}
    geo = (spec["batch"], spec["n_kv"], spec["max_tokens"], spec["n_words"])
    for kind, t0, x in spec["windows"]:
        rec, alpha = O.cache_records(img, *geo, spec["b"], spec["h"], kind, t0, x.shape[0])
        st, err = code_check(x, rec, alpha, spec["enc"][kind], spec["bits"][kind], spec["scales"][kind])
        st["kind"] = kind
        res["stats"].append(st)
        if err:
            res["error"] = f"b {spec['b']} head {spec['h']} kind {kind}: {err}"
            return res
    if spec.get("q") is not None:
        hh = []
        for kind in (0, 1):
            rec, alpha = O.cache_records(img, *geo, spec["b"], spec["h"], kind, 0, spec["n_ctx"])
            bits = np.asarray(spec["bits"][kind]).astype(np.int64)
            codes = O.unpack_records(rec, bits)
            hh.append(O.dequantize_f32(codes, alpha, spec["scales"][kind], bits))
        q = np.asarray(spec["q"], np.float64)
        res["out"] = O.decode_attention(q, hh[0][None], hh[1][None], spec["basis"][0][None], spec["basis"][1][None],
                                        q.shape[0])
    return res
