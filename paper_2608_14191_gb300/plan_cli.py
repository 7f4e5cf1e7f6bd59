"""Command-line planner: calibration arrays in, plan file out (host only, no GPU).

    python -m paper_2608_14191_gb300.plan_cli calib.npz plan.aatc --bits 2.75 [--bits-v B]
        [--var-only] [--global --protect 3] [--b-max 8]

calib.npz holds `k` and `v` (fp32 [L][H_kv][N][128] calibration keys / values) and optionally `q`
(fp32 [L][H_q][N_q][128] calibration queries; without it the key weights are 1).  The planner is
the library's (Sec. 5 Steps 1-2: second moment, eigenbasis, weights, integer reverse
water-filling, P99 scales); --global replaces the per-stream budgets with one pool per kind over
all layers (the first --protect layers planned per stream).  Prints the width histogram of every
stream and the code bits per token.
"""
from __future__ import annotations

import argparse
import sys

import numpy as np

from . import allocate_global, calibrate, dims, save_plan


def plan_from_arrays(k: np.ndarray, v: np.ndarray, q: np.ndarray | None, bits_k: float, bits_v: float,
                     var_only: bool = False, global_pool: bool = False, n_protect: int = 3, b_max: int = 8):
    """(dims, dict(basis, bits, scales)) for calibration arrays as the module docstring describes."""
    if k.ndim != 4 or v.shape != k.shape or k.shape[-1] != 128:
        raise ValueError("k and v must both be [L][H_kv][N][128]")
    L, H = k.shape[0], k.shape[1]
    n_q = H if q is None else q.shape[1]
    if q is not None and (q.ndim != 4 or q.shape[0] != L or q.shape[-1] != 128):
        raise ValueError("q must be [L][H_q][N_q][128]")
    dm = dims(L, H, n_q, b_max=b_max)
    cal = calibrate(dm, k, v, q, bits_k, bits_v, var_only=var_only)
    bits = cal["bits"]
    if global_pool:
        bits = allocate_global(dm, cal["sigma2"], cal["weights"], bits_k, bits_v, n_protect=n_protect)
    return dm, {"basis": cal["basis"], "bits": bits, "scales": cal["scales"]}


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description="calibrate an AATC plan and write it to a plan file")
    ap.add_argument("calib", help=".npz with k, v [L][H_kv][N][128] and optionally q [L][H_q][N_q][128]")
    ap.add_argument("out", help="plan file to write")
    ap.add_argument("--bits", type=float, required=True, help="average code bits per key channel")
    ap.add_argument("--bits-v", type=float, default=None, help="average bits per value channel (default: --bits)")
    ap.add_argument("--var-only", action="store_true", help="variance-only weights (w = 1)")
    ap.add_argument("--global", dest="global_pool", action="store_true", help="one pool per kind over all layers")
    ap.add_argument("--protect", type=int, default=3, help="layers planned per stream under --global")
    ap.add_argument("--b-max", type=int, default=8, help="widest channel (8 for device plans, up to 16)")
    a = ap.parse_args(argv)
    with np.load(a.calib) as z:
        k = np.ascontiguousarray(z["k"], dtype=np.float32)
        v = np.ascontiguousarray(z["v"], dtype=np.float32)
        q = np.ascontiguousarray(z["q"], dtype=np.float32) if "q" in z.files else None
    bits_v = a.bits if a.bits_v is None else a.bits_v
    dm, p = plan_from_arrays(k, v, q, a.bits, bits_v, a.var_only, a.global_pool, a.protect, a.b_max)
    save_plan(a.out, dm, p["basis"], p["bits"], p["scales"])
    b = p["bits"].astype(np.int64)
    for layer in range(dm.n_layers):
        for h in range(dm.n_kv_heads):
            for kind, name in ((0, "K"), (1, "V")):
                hist = np.bincount(b[layer, h, kind], minlength=dm.b_max + 1)
                print(f"layer {layer} kv-head {h} {name}: {int(b[layer, h, kind].sum())} bits, widths 0..{dm.b_max}: "
                      f"{hist.tolist()}")
    print(f"wrote {a.out}: {dm.n_layers} layers x {dm.n_kv_heads} kv-heads, "
          f"{b.sum() / (dm.n_layers * dm.n_kv_heads):.1f} code bits per token and kv-head (K + V, layer mean)")
    return 0


if __name__ == "__main__":
    sys.exit(main())
