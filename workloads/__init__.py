"""Seeded synthetic KV-cache workloads shared by the oracle, the tests and the bench.

This module holds only the *input* model, none of the compression method's
arithmetic.  It stands in for the paper's Llama-3.1-8B / Qwen-2.5-7B caches and
calibration corpora (Section 6 of the paper), which are not available here.

Input model (per layer l, kv-head h and kind K|V, called a *stream*):
  * U  : a Haar-random orthogonal 128x128 matrix (QR of a Gaussian, column signs
         taken from diag(R)),
  * lam: power-law spectrum lam_i = i**-1.5, i = 1..128 (not renormalised),
  * x = U diag(lam)^(1/2) z with z ~ N(0, I); keys additionally get 4 outlier
    coordinates (seeded per layer and head) multiplied by 8 after the Gaussian
    draw; everything is rounded to bf16.
Decode and calibration queries are N(0, I) bf16 by default; an anisotropic query
model N(0, V diag(i^-1) V^T) exists to exercise the attention-aware weights.

Seeds: base = 1000 + config number (1..5); every random draw comes from
numpy.random.SeedSequence(base, spawn_key=(layer, head, kind, purpose)).
Bulk cache data for the GPU is drawn with torch on the target device from a
seed taken from the same key, so host copies of it are exact inputs for the
oracle (the data is an input: generator determinism never affects parity).
"""
from __future__ import annotations

import dataclasses
import numpy as np

D = 128                  # head_dim
N_CALIB = 4096           # calibration vectors per stream and queries per q-head
N_OUTLIERS = 4
OUTLIER_GAIN = 8.0
KIND_K, KIND_V = 0, 1
_PURPOSE = {"basis": 0, "calib": 1, "data": 2, "query": 3, "calib_query": 4, "query_model": 5,
            "hidden_model": 6, "hidden_calib": 7, "hidden_data": 8, "weight": 9}


@dataclasses.dataclass(frozen=True)
class Config:
    number: int          # 1..5, the order in which the workloads are listed
    name: str
    n_layers: int
    n_kv_heads: int
    n_q_heads: int
    batch: int
    n_ctx: int
    avg_bits: tuple
    decode_steps: int
    workload: str

    @property
    def seed(self) -> int:
        return 1000 + self.number

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads


CONFIGS = {
    "tiny": Config(1, "tiny", 1, 1, 4, 1, 512, (2.75,), 1,
                   "encode 512 tokens, one decode step"),
    "llama_layer": Config(2, "llama_layer", 1, 8, 32, 1, 32768, (2.75,), 256,
                          "Llama-3.1-8B-shaped layer: encode 32768 tokens x 8 kv-heads, "
                          "then 256 decode steps with random bf16 queries"),
    "qwen": Config(3, "qwen", 1, 4, 28, 16, 8192, (2.75,), 1,
                   "Qwen-2.5-7B-shaped layer: prefill-encode 16 x 8192 tokens, one batched decode"),
    "llama_stack": Config(4, "llama_stack", 32, 8, 32, 1, 131072, (2.75,), 1,
                          "Llama-3.1-8B-shaped 32-layer stack at 131072 tokens: one decode step "
                          "through all layers"),
    "sweep": Config(5, "sweep", 1, 8, 32, 4, 32768, (1.5, 2.0, 2.75, 4.0), 1,
                    "Llama shape, batch 4 x 32768 tokens, encode + decode at 1.5/2/2.75/4 bits"),
}


def _rng(seed: int, layer: int, head: int, kind: int, purpose: str) -> np.random.Generator:
    ss = np.random.SeedSequence(seed, spawn_key=(layer, head, kind, _PURPOSE[purpose]))
    return np.random.default_rng(ss)


def torch_seed(seed: int, layer: int, head: int, kind: int, purpose: str) -> int:
    """A 63-bit integer seed for torch generators, derived from the same key."""
    ss = np.random.SeedSequence(seed, spawn_key=(layer, head, kind, _PURPOSE[purpose]))
    return int(ss.generate_state(1, dtype=np.uint64)[0]) & ((1 << 63) - 1)


def power_law(d: int = D) -> np.ndarray:
    return np.arange(1, d + 1, dtype=np.float64) ** -1.5


def haar_orthogonal(rng: np.random.Generator, d: int = D) -> np.ndarray:
    g = rng.standard_normal((d, d))
    q, r = np.linalg.qr(g)
    return q * np.sign(np.diag(r))[None, :]


@dataclasses.dataclass(frozen=True)
class StreamModel:
    """Covariance model of one stream: x = mix @ z, then outlier coordinates x gain."""
    mix: np.ndarray          # (128, 128) = U diag(sqrt(lam))
    outliers: np.ndarray     # int indices into the 128 coordinates (empty for values)
    gain: float = OUTLIER_GAIN

    def transform(self, z: np.ndarray) -> np.ndarray:
        x = z @ self.mix.T
        if len(self.outliers):
            x[:, self.outliers] *= self.gain
        return x


def stream_model(seed: int, layer: int, head: int, kind: int) -> StreamModel:
    rng = _rng(seed, layer, head, kind, "basis")
    u = haar_orthogonal(rng)
    mix = u * np.sqrt(power_law())[None, :]
    if kind == KIND_K:
        # Outlier coordinates are per (layer, kv-head); drawn from the key stream's basis rng.
        idx = np.sort(rng.choice(D, N_OUTLIERS, replace=False))
    else:
        idx = np.zeros(0, dtype=np.int64)
    return StreamModel(mix=mix, outliers=idx)


def to_bf16(x):
    """Round float data to bf16 (round-to-nearest-even on the float32 value); returns float32
    numpy values.  Done on the float32 bit pattern: add 0x7FFF plus the lowest kept bit, then
    clear the low 16 bits (the same values as torch's float32 -> bfloat16 cast for finite
    inputs, which tests/test_workloads.py checks)."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(f.shape)


def calibration_vectors(cfg: Config, layer: int, head: int, kind: int, n: int = N_CALIB) -> np.ndarray:
    """(n, 128) float32 array of bf16-exact calibration vectors for one stream."""
    m = stream_model(cfg.seed, layer, head, kind)
    z = _rng(cfg.seed, layer, head, kind, "calib").standard_normal((n, D))
    return to_bf16(m.transform(z))


def query_model(cfg: Config, layer: int, q_head: int, anisotropic: bool) -> np.ndarray:
    """(128, 128) mixing matrix A of the query model q = A z (identity if isotropic)."""
    if not anisotropic:
        return np.eye(D)
    rng = _rng(cfg.seed, layer, q_head, 0, "query_model")
    v = haar_orthogonal(rng)
    return v * np.sqrt(1.0 / np.arange(1, D + 1))[None, :]


def calibration_queries(cfg: Config, layer: int, q_head: int, n: int = N_CALIB,
                        anisotropic: bool = False) -> np.ndarray:
    z = _rng(cfg.seed, layer, q_head, 0, "calib_query").standard_normal((n, D))
    return to_bf16(z @ query_model(cfg, layer, q_head, anisotropic).T)


def layer_calibration(cfg: Config, layer: int, anisotropic_queries: bool = False, n: int = N_CALIB):
    """Calibration inputs for one layer in the C-ABI layouts.

    Returns (calib_k, calib_v, calib_q) with shapes (H_kv, n, 128), (H_kv, n, 128),
    (H_q, n, 128), all float32 holding bf16-exact values.
    """
    ck = np.stack([calibration_vectors(cfg, layer, h, KIND_K, n) for h in range(cfg.n_kv_heads)])
    cv = np.stack([calibration_vectors(cfg, layer, h, KIND_V, n) for h in range(cfg.n_kv_heads)])
    cq = np.stack([calibration_queries(cfg, layer, j, n, anisotropic_queries)
                   for j in range(cfg.n_q_heads)])
    return ck, cv, cq


def kv_host(cfg: Config, layer: int, batch: int, n_tokens: int, offset_seed: int = 0):
    """Host (numpy) K, V of shape (batch, n_tokens, H_kv, 128), bf16-exact float32.

    Used for small cases; large cases use :func:`kv_device`.
    """
    k = np.empty((batch, n_tokens, cfg.n_kv_heads, D), np.float32)
    v = np.empty_like(k)
    for h in range(cfg.n_kv_heads):
        for kind, out in ((KIND_K, k), (KIND_V, v)):
            m = stream_model(cfg.seed, layer, h, kind)
            rng = _rng(cfg.seed + offset_seed, layer, h, kind, "data")
            z = rng.standard_normal((batch * n_tokens, D))
            out[:, :, h, :] = to_bf16(m.transform(z)).reshape(batch, n_tokens, D)
    return k, v


def kv_device(cfg: Config, layer: int, batch: int, n_tokens: int, device, offset_seed: int = 0):
    """Device bf16 K, V of shape (batch, n_tokens, H_kv, 128), drawn with torch on `device`."""
    import torch
    k = torch.empty((batch, n_tokens, cfg.n_kv_heads, D), dtype=torch.bfloat16, device=device)
    v = torch.empty_like(k)
    for h in range(cfg.n_kv_heads):
        for kind, out in ((KIND_K, k), (KIND_V, v)):
            m = stream_model(cfg.seed, layer, h, kind)
            g = torch.Generator(device=device)
            g.manual_seed(torch_seed(cfg.seed + offset_seed, layer, h, kind, "data"))
            mix = torch.from_numpy(m.mix.astype(np.float32)).to(device)
            chunk = 1 << 20
            total = batch * n_tokens
            flat = out.view(total, cfg.n_kv_heads, D)
            for s in range(0, total, chunk):
                e = min(total, s + chunk)
                z = torch.randn((e - s, D), generator=g, device=device, dtype=torch.float32)
                x = z @ mix.T
                if len(m.outliers):
                    idx = torch.from_numpy(m.outliers).to(device)
                    x[:, idx] *= m.gain
                flat[s:e, h, :] = x.to(torch.bfloat16)
    return k, v


def queries_device(cfg: Config, layer: int, batch: int, steps: int, device, peaky: float = 1.0):
    """Device bf16 decode queries of shape (steps, batch, H_q, 128), N(0, peaky^2 I)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(torch_seed(cfg.seed, layer, 0, 0, "query"))
    q = torch.randn((steps, batch, cfg.n_q_heads, D), generator=g, device=device) * peaky
    return q.to(torch.bfloat16)


def queries_host(cfg: Config, layer: int, batch: int, steps: int, peaky: float = 1.0) -> np.ndarray:
    rng = _rng(cfg.seed, layer, 0, 0, "query")
    return to_bf16(rng.standard_normal((steps, batch, cfg.n_q_heads, D)) * peaky)


# ----------------------------------------------------------------------------
# Hidden states and projection weights (the transform from model weights, Sec. 5 Step 1)
# ----------------------------------------------------------------------------
# Stand-in for a layer's input activations X (T x d_model) and its key / value projection
# W (d_model x n_kv*128), which the paper takes from the model checkpoints:
#   * x = (z * sqrt(lam)) @ M / sqrt(d_model) with z ~ N(0, I), lam_i = i**-1.0 over d_model
#     coordinates, M a Gaussian d_model x d_model matrix (anisotropic, correlated activations),
#     plus 4 outlier coordinates x 20 (the heavy channels of transformer hidden states);
#   * W ~ N(0, 1/d_model), one matrix per (layer, kind), columns head-major (head h owns
#     columns 128h .. 128h + 127).
N_HIDDEN_OUTLIERS = 4
HIDDEN_OUTLIER_GAIN = 20.0


def hidden_model(seed: int, layer: int, d_model: int):
    """(mix (d_model x d_model), outlier indices) of the hidden-state model of one layer."""
    rng = _rng(seed, layer, 0, 0, "hidden_model")
    lam = np.arange(1, d_model + 1, dtype=np.float64) ** -1.0
    mix = (np.sqrt(lam)[:, None] * rng.standard_normal((d_model, d_model))) / np.sqrt(d_model)
    idx = np.sort(rng.choice(d_model, N_HIDDEN_OUTLIERS, replace=False))
    return mix, idx


def hidden_states(seed: int, layer: int, d_model: int, n: int, purpose: str = "hidden_calib") -> np.ndarray:
    """(n, d_model) float32 bf16-exact hidden states of one layer (host)."""
    mix, idx = hidden_model(seed, layer, d_model)
    z = _rng(seed, layer, 0, 0, purpose).standard_normal((n, d_model)).astype(np.float32)
    x = z @ mix.astype(np.float32)
    x[:, idx] *= HIDDEN_OUTLIER_GAIN
    return to_bf16(x)


def hidden_states_device(seed: int, layer: int, d_model: int, batch: int, n_tokens: int, device):
    """bf16 [batch][n_tokens][d_model] hidden states drawn on the device (same model, torch
    generator seeded from the (layer, "hidden_data") key)."""
    import torch
    mix, idx = hidden_model(seed, layer, d_model)
    gen = torch.Generator(device=device)
    gen.manual_seed(torch_seed(seed, layer, 0, 0, "hidden_data"))
    m = torch.from_numpy(mix.astype(np.float32)).to(device)
    x = torch.empty((batch * n_tokens, d_model), dtype=torch.bfloat16, device=device)
    for r0 in range(0, batch * n_tokens, 8192):
        r1 = min(batch * n_tokens, r0 + 8192)
        z = torch.randn((r1 - r0, d_model), generator=gen, device=device, dtype=torch.float32)
        y = z @ m
        y[:, torch.from_numpy(idx).to(device)] *= HIDDEN_OUTLIER_GAIN
        x[r0:r1] = y.to(torch.bfloat16)
    return x.view(batch, n_tokens, d_model)


def projection_weight(seed: int, layer: int, kind: int, d_model: int, n_kv: int) -> np.ndarray:
    """(d_model, n_kv * 128) float32 bf16-exact key (kind 0) or value (kind 1) projection."""
    rng = _rng(seed, layer, 0, kind, "weight")
    return to_bf16(rng.standard_normal((d_model, n_kv * D)) / np.sqrt(d_model))
