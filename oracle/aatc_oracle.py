"""AATC oracle: a plain, slow, fp64 CPU restatement of the paper's method.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / reference leg of ``bench.py`` may import this module.  It shares
no code with the CUDA library (``paper_2608_14191_gb300``) and imports nothing
from it; the only shared module is ``workloads`` (seeded inputs, no method
arithmetic).

Every function cites the passage of arxiv 2608.14191 ("KV Cache Compression
Through the Lens of Transform Coding") that it follows.  Floating point is fp64
except :func:`dequantize_f32`, which spells out the two fp32 multiplies that
define the stored-code reconstruction so that the GPU's can be checked bit for
bit.

Pins (tests/test_oracle_pins.py) tie each function to something other than
itself: the transform round trip (Sec. 3.1), the reverse water-filling closed
form (Eq. bit-allocation, Sec. 3.1), brute force over integer allocations at d=4
(Eq. waterfilling-keys), a Monte Carlo check of Theorem 1, the whitening-SVD /
PCA equivalence (Appendix, Proposition), the quantizer error bound
(Def. uniform-quant), library SDPA for decode, hand-computed small cases and
the compression ratio the paper prints (Sec. 6.1); the transform from the model
weights (:func:`whitening_transform`, tests/test_whitening.py) is pinned by
W = A B, A^T Sigma_X A = S and both statements of the appendix Proposition.
Head-group bases (:func:`plan_head_group`, :func:`decode_attention_head_group`,
tests/test_head_groups.py) are pinned by the reduction to the per-head plan and
decode at one head per group, plain attention per query head when the group
coefficients are exact, the split of an exactly block-diagonal second moment
into the heads' own eigenbases, the budget identity, and the transform-coding
gain of one group transform over separate heads for correlated heads.

parity unpinned: the packed record bit layout (:func:`record_entries`,
:func:`pack_records`, :func:`cache_records`) is defined by this library, not by the
paper, which prints no worked encoding.  It is pinned only by the round trip
unpack(pack(c)) == c, the record-size identity (352 code bits per token and stream
at 2.75 bits, i.e. the paper's 16/2.75 = 5.82x, in exactly 11 words) and
hand-computed packed words.
"""
from __future__ import annotations

import math
import numpy as np

D = 128
TILE = 128          # tokens per word-planar tile of the packed cache


# ----------------------------------------------------------------------------
# Offline calibration (Sec. 5, Algorithm 1 calibration half, Appendix A.x)
# ----------------------------------------------------------------------------

def second_moment(x: np.ndarray) -> np.ndarray:
    """Uncentered empirical second moment C = X^T X / N (Sec. 5 Step 1, Sigma_X = X^T X / T)."""
    x = np.asarray(x, dtype=np.float64)
    return x.T @ x / x.shape[0]


def canonical_sign(vectors: np.ndarray) -> np.ndarray:
    """Flip each column so that its largest-magnitude entry (lowest index on ties) is positive.

    The paper leaves eigenvector signs open; this is the library's convention.
    """
    v = np.array(vectors, dtype=np.float64, copy=True)
    for j in range(v.shape[1]):
        i = int(np.argmax(np.abs(v[:, j])))
        if v[i, j] < 0:
            v[:, j] = -v[:, j]
    return v


def eigenbasis(c: np.ndarray):
    """Eigen-decomposition C = U diag(lam) U^T, eigenvalues descending (Sec. 3.1, KLT;
    Appendix Proposition: the PCA of K = XW equals the whitening-SVD transform)."""
    lam, vec = np.linalg.eigh(np.asarray(c, dtype=np.float64))
    order = np.argsort(-lam, kind="stable")
    return lam[order], canonical_sign(vec[:, order])


def whitening_transform(x_calib: np.ndarray, w: np.ndarray):
    """Whitening-based feature decorrelation from the model weights (Sec. 5 Step 1, Eq.
    AB-factorization), in the paper's order:
      Sigma_X = X^T X / T;  Sigma_X = L L^T (Cholesky);  W~ = L^T W;  W~ = U S P^T (reduced SVD);
      A = L^-T U sqrt(S);  B = sqrt(S) P^T,  so that W = A B and H = X A is cached.
    x_calib: (T, d_model) calibration activations; w: (d_model, d) one head's projection.
    Singular vectors are sign-canonical in P (largest |entry| positive), U flipped alike, so A B
    is unchanged.  Returns dict(A (d_model, d), B (d, d), S (d,), P (d, d), U, L)."""
    x = np.asarray(x_calib, dtype=np.float64)
    w = np.asarray(w, dtype=np.float64)
    sigma_x = x.T @ x / x.shape[0]
    l_chol = np.linalg.cholesky(sigma_x)
    w_tilde = l_chol.T @ w
    u, s, pt = np.linalg.svd(w_tilde, full_matrices=False)
    p_mat = pt.T
    cols = np.arange(p_mat.shape[1])
    flip = np.where(p_mat[np.argmax(np.abs(p_mat), axis=0), cols] < 0, -1.0, 1.0)   # as canonical_sign
    p_mat = p_mat * flip[None, :]
    u = u * flip[None, :]
    a = np.linalg.solve(l_chol.T, u) * np.sqrt(s)[None, :]
    b = np.sqrt(s)[:, None] * p_mat.T
    return {"A": a, "B": b, "S": s, "P": p_mat, "U": u, "L": l_chol}


def hidden_encode_operand(a: np.ndarray, s: np.ndarray) -> np.ndarray:
    """A sqrt(S) = W P: the encode matrix of the cached coefficients with each column rescaled
    by sqrt(S_c).  Per-column positive scaling leaves the allocation and the codes unchanged
    (Eq. AB-factorization with the quantizer of Sec. 5: s_c and h_c scale alike), so caching
    x A sqrt(S) instead of x A gives the same codes as the PCA coefficients of k = x W."""
    return np.asarray(a, dtype=np.float64) * np.sqrt(np.asarray(s, dtype=np.float64))[None, :]


def channel_variance(encode_basis: np.ndarray, x: np.ndarray) -> np.ndarray:
    """sigma_c^2 = mean over calibration of h_c^2 with h = x A (Alg. 1 calibration, 'record latent
    variance'; uncentered because the source is zero-mean, Sec. 3.1)."""
    h = np.asarray(x, np.float64) @ encode_basis
    return np.mean(h * h, axis=0)


def key_weights(recon_rows: np.ndarray, queries_by_head) -> np.ndarray:
    """w^K_c = sum over the query heads of the GQA group of (1/T) sum_i (B_c . q_i)^2
    (Eq. waterfilling-keys; GQA remark in the appendix derivation).  ``recon_rows`` is B
    (channel c reconstructs along row B_c); for an orthonormal basis B = U^T."""
    b = np.asarray(recon_rows, np.float64)
    w = np.zeros(b.shape[0])
    for q in queries_by_head:
        proj = np.asarray(q, np.float64) @ b.T          # (T, channels)
        w += np.mean(proj * proj, axis=0)
    return w


def value_weights(recon_rows: np.ndarray, w_o: np.ndarray | None = None) -> np.ndarray:
    """w^V_c = ||(B^V W_O)_c||^2 (Sec. 5 Step 2, values).  The decode path has no output
    projection (Alg. 1 output line), so W_O = I by default and w^V_c = ||B_c||^2."""
    b = np.asarray(recon_rows, np.float64)
    m = b if w_o is None else b @ np.asarray(w_o, np.float64)
    return np.sum(m * m, axis=1)


def allocation_objective(g: np.ndarray, bits: np.ndarray) -> float:
    """Weighted distortion surrogate sum_c g_c 2^(-2 b_c) (Eq. waterfilling-keys objective with
    g_c = w_c sigma_c^2; the common constant gamma of Eq. noise-model drops out)."""
    return float(np.sum(np.asarray(g, np.float64) * np.exp2(-2.0 * np.asarray(bits, np.float64))))


def greedy_allocation(g: np.ndarray, budget: int, b_max: int) -> np.ndarray:
    """Integer reverse water-filling: minimise sum_c g_c 4^(-b_c) s.t. sum b_c <= budget,
    b_c in {0..b_max} (Eq. waterfilling-keys; Remark 'Zero-bit dimensions').

    The objective is separable with convex, decreasing per-channel terms, so handing out
    one bit at a time to the channel whose term drops the most is exactly optimal.  The
    drop for channel c at b_c bits is (3/4) g_c 4^(-b_c); the 3/4 is common and omitted.
    Ties go to the lowest channel index.
    """
    g = np.asarray(g, np.float64)
    bits = np.zeros(len(g), dtype=np.int64)
    for _ in range(int(budget)):
        gain = np.where(bits < b_max, g * np.exp2(-2.0 * bits), -np.inf)
        c = int(np.argmax(gain))
        if not np.isfinite(gain[c]):
            break
        bits[c] += 1
    return bits


def continuous_allocation(g: np.ndarray, budget: float, b_max: float = np.inf):
    """Continuous reverse water-filling (Eq. bit-allocation, weighted form of Sec. 5 Step 2):
    b_c = clip(1/2 log2(g_c / theta), 0, b_max) with the water level theta chosen so that
    sum_c b_c = budget.  Returns (bits, theta)."""
    g = np.asarray(g, np.float64)

    def total(log_theta):
        return float(np.sum(np.clip(0.5 * (np.log2(g) - log_theta), 0.0, b_max)))

    lo, hi = math.log2(g.min()) - 2 * 64, math.log2(g.max())
    for _ in range(400):
        mid = 0.5 * (lo + hi)
        if total(mid) > budget:
            lo = mid
        else:
            hi = mid
    theta_log = 0.5 * (lo + hi)
    return np.clip(0.5 * (np.log2(g) - theta_log), 0.0, b_max), 2.0 ** theta_log


def global_allocation(sigma2: np.ndarray, weights: np.ndarray, avg_bits_k: float, avg_bits_v: float,
                      n_protect: int = 3, b_max: int = 8) -> np.ndarray:
    """Global cross-layer allocation (Eq. waterfilling-keys and its value twin, both summed over
    layers; Algorithm 1, global reverse water-filling over every (layer, channel) pair; the
    AATC experimental-setup paragraph for the protected layers and the normalisation).

    sigma2, weights: [L][H][2][d] (kind 0 keys, 1 values), channels in storage order.
    Per kind: layers l < n_protect are allocated per stream with the average budget (values) or
    one bit per channel more (keys, capped at b_max d); the rest of the kind's total budget
    avg_bits * d * L * H is water-filled over every channel of the other layers at once, with
    sigma^2 and w each divided by the layer's own 95th percentile over its channels (all kv-heads).
    b_max: 8 for what a device plan holds; the paper allows 16, which the planner also takes.
    """
    sigma2 = np.asarray(sigma2, np.float64)
    weights = np.asarray(weights, np.float64)
    L, H, _, d = sigma2.shape
    bits = np.zeros(sigma2.shape, dtype=np.int64)
    np_ = min(n_protect, L)
    for kind, avg in ((0, avg_bits_k), (1, avg_bits_v)):
        per_stream = int(round(avg * d))
        prot = min(per_stream + (d if kind == 0 else 0), b_max * d)
        for l in range(np_):
            for h in range(H):
                bits[l, h, kind] = greedy_allocation(weights[l, h, kind] * sigma2[l, h, kind], prot, b_max)
        rest = per_stream * L * H - prot * np_ * H
        if rest < 0 or rest > b_max * d * (L - np_) * H:
            raise ValueError("the protected layers and the pool do not fit the total budget")
        if np_ == L:
            continue
        g = []
        for l in range(np_, L):
            ps = percentile_linear(sigma2[l, :, kind].ravel(), 95.0)
            pw = percentile_linear(weights[l, :, kind].ravel(), 95.0)
            ps = ps if ps > 0 else 1.0
            pw = pw if pw > 0 else 1.0
            g.append((sigma2[l, :, kind] / ps) * (weights[l, :, kind] / pw))
        pooled = greedy_allocation(np.concatenate([x.ravel() for x in g]), rest, b_max)
        bits[np_:, :, kind] = pooled.reshape(L - np_, H, d)
    return bits


def percentile_linear(values: np.ndarray, p: float) -> float:
    """Percentile with linear interpolation at rank (p/100)(N-1) of the sorted sample."""
    a = np.sort(np.asarray(values, np.float64))
    pos = (p / 100.0) * (len(a) - 1)
    lo = int(math.floor(pos))
    hi = min(lo + 1, len(a) - 1)
    return float(a[lo] + (pos - lo) * (a[hi] - a[lo]))


def channel_scales(encode_basis: np.ndarray, x: np.ndarray, p: float = 99.0) -> np.ndarray:
    """s_c = 99th percentile of |h_c| over the calibration tokens (Sec. 5, 'The right scaling')."""
    h = np.abs(np.asarray(x, np.float64) @ encode_basis)
    return np.array([percentile_linear(h[:, c], p) for c in range(h.shape[1])])


def plan_stream(x_calib: np.ndarray, avg_bits: float, b_max: int = 8, queries_by_head=None,
                weights: str = "aatc"):
    """Calibrate one stream (one layer, kv-head and K|V): Algorithm 1 calibration half with the
    PCA eigenbasis standing in for the whitening-SVD transform (Appendix Proposition).

    weights: 'aatc' (keys: query weights if queries_by_head is given; values: W_O = I) or
    'var' (AATC var-only: w = 1, Sec. 6).
    Channels are stored in descending order of g_c = w_c sigma_c^2 (stable), which makes the
    bit widths non-increasing along storage order.
    """
    c = second_moment(x_calib)
    lam, u = eigenbasis(c)
    if weights == "var":
        w = np.ones(D)
    elif queries_by_head is not None:
        w = key_weights(u.T, queries_by_head)
    else:
        w = value_weights(u.T)
    g = w * lam
    order = np.argsort(-g, kind="stable")
    u, lam, w, g = u[:, order], lam[order], w[order], g[order]
    budget = int(round(avg_bits * D))
    bits = greedy_allocation(g, budget, b_max)
    scales = channel_scales(u, x_calib)
    return {"basis": u, "bits": bits, "scales": scales, "sigma2": lam, "weights": w, "g": g}


# ----------------------------------------------------------------------------
# Online encode (Algorithm 1 inference half: project, quantize, append)
# ----------------------------------------------------------------------------

def token_scale(h: np.ndarray, scales: np.ndarray, bits: np.ndarray) -> np.ndarray:
    """alpha_t = max_c |h_c / s_c| over the retained channels (b_c >= 1) (Sec. 5, token scale)."""
    keep = np.asarray(bits) > 0
    return np.max(np.abs(h[:, keep]) / np.asarray(scales, np.float64)[keep], axis=1)


def quantize(h: np.ndarray, alpha: np.ndarray, scales: np.ndarray, bits: np.ndarray):
    """Symmetric uniform quantizer of Sec. 5: Delta = 2 alpha s_c / 2^b_c,
    code = clamp(floor(h/Delta + 1/2), -2^(b-1), 2^(b-1) - 1).  Channels with b_c = 0 are
    dropped (code 0).  Returns (codes, t = h/Delta) with t = 0 where alpha = 0."""
    h = np.asarray(h, np.float64)
    b = np.asarray(bits, np.int64)
    s = np.asarray(scales, np.float64)
    keep = b > 0
    codes = np.zeros(h.shape, dtype=np.int64)
    t = np.zeros(h.shape)
    delta = 2.0 * alpha[:, None] * s[None, keep] / np.exp2(b[keep])[None, :]
    with np.errstate(divide="ignore", invalid="ignore"):
        tk = np.where(delta > 0, h[:, keep] / np.where(delta > 0, delta, 1.0), 0.0)
    lo = -np.exp2(b[keep] - 1)
    hi = np.exp2(b[keep] - 1) - 1
    codes[:, keep] = np.clip(np.floor(tk + 0.5), lo, hi).astype(np.int64)
    t[:, keep] = tk
    return codes, t


def dequantize(codes: np.ndarray, alpha: np.ndarray, scales: np.ndarray, bits: np.ndarray):
    """dqtz(c) = Delta c (Sec. 5), fp64."""
    b = np.asarray(bits, np.int64)
    delta = 2.0 * alpha[:, None] * np.asarray(scales, np.float64)[None, :] / np.exp2(b)[None, :]
    return np.where(b[None, :] > 0, codes * delta, 0.0)


def encode_stream(x: np.ndarray, encode_basis: np.ndarray, bits: np.ndarray, scales: np.ndarray):
    """Project h = x A (Alg. 1 'Project'), per-token scale, quantize (Alg. 1 'Append qtz(h)').

    Returns (codes (n,128) int, alpha (n,) fp64, t (n,128) = h/Delta)."""
    h = np.asarray(x, np.float64) @ np.asarray(encode_basis, np.float64)
    alpha = token_scale(h, scales, bits)
    codes, t = quantize(h, alpha, scales, bits)
    return codes, alpha, t


def dequantize_f32(codes: np.ndarray, alpha_f32: np.ndarray, scales_f32: np.ndarray,
                   bits: np.ndarray) -> np.ndarray:
    """Stored-code reconstruction in fp32, two correctly rounded multiplies in this order:
    f_c = s_c 2^(1-b_c) (exact), Delta = fl32(alpha f_c), h_hat = fl32(code Delta)
    (Sec. 5 dqtz with Delta = 2 alpha s_c / 2^b_c)."""
    b = np.asarray(bits, np.int64)
    f = (np.asarray(scales_f32, np.float32) * np.exp2(1 - b).astype(np.float32)).astype(np.float32)
    delta = (np.asarray(alpha_f32, np.float32)[:, None] * f[None, :]).astype(np.float32)
    out = (np.asarray(codes).astype(np.float32) * delta).astype(np.float32)
    return np.where(b[None, :] > 0, out, np.float32(0.0)).astype(np.float32)


# ----------------------------------------------------------------------------
# Packed layout (library-defined; the paper prints none)
#
# Each stored code is u = code + 2^(b-1) (offset binary, b bits).  The record of one token
# and stream splits u into base-4 digits and single top bits, grouped by significance:
#   D2 = for k = 0..7: digit k (bits 2k, 2k+1) of every channel with b >= 2k+2 (b up to 16)
#   D1 = the top bit (bit b-1) of every odd-width channel, in channel order
# Channels are in storage order (widths non-increasing), so each D2 layer is a prefix.  If |D2| is not a multiple of 16, its last |D2| mod 16
# entries move to the end of D1 as two single bits each.  Record words: the D2 entries at
# 16 per word (entry i at bits 2(i mod 16)), then the D1 entries at 32 per word (entry j at
# bit j mod 32), then zero words up to W.
# ----------------------------------------------------------------------------

def record_entries(bits: np.ndarray):
    """(D2, D1): lists of (channel, bit shift) entries of one stream's record."""
    b = [int(x) for x in bits]
    assert max(b, default=0) <= 16
    d2 = []
    for k in range(8):
        d2 += [(c, 2 * k) for c in range(len(b)) if b[c] >= 2 * k + 2]
    d1 = [(c, b[c] - 1) for c in range(len(b)) if b[c] % 2 == 1]
    r = len(d2) % 16
    if r:
        moved = d2[len(d2) - r:]
        d2 = d2[:len(d2) - r]
        for (c, sh) in moved:
            d1 += [(c, sh), (c, sh + 1)]
    return d2, d1


def stream_words(bits: np.ndarray) -> int:
    d2, d1 = record_entries(bits)
    return len(d2) // 16 + (len(d1) + 31) // 32


def record_words(bits_per_stream) -> int:
    """Words per record: W = max over streams, at least 1."""
    return max(1, max(stream_words(b) for b in bits_per_stream))


def pack_records(codes: np.ndarray, bits: np.ndarray, n_words: int) -> np.ndarray:
    """codes (n, 128) signed -> (n, n_words) uint32 records (token-major, before any interleave)."""
    b = np.asarray(bits, np.int64)
    u = np.where(b[None, :] > 0, codes + np.where(b > 0, 2 ** np.maximum(b - 1, 0), 0)[None, :], 0).astype(np.uint64)
    assert np.all(u < np.where(b > 0, 2 ** b, 1)[None, :])
    d2, d1 = record_entries(b)
    words = np.zeros((codes.shape[0], n_words), dtype=np.uint64)
    for i, (c, sh) in enumerate(d2):
        words[:, i // 16] |= ((u[:, c] >> np.uint64(sh)) & np.uint64(3)) << np.uint64(2 * (i % 16))
    base = len(d2) // 16
    for j, (c, sh) in enumerate(d1):
        words[:, base + j // 32] |= ((u[:, c] >> np.uint64(sh)) & np.uint64(1)) << np.uint64(j % 32)
    assert base + (len(d1) + 31) // 32 <= n_words
    return words.astype(np.uint32)


def unpack_records(words: np.ndarray, bits: np.ndarray) -> np.ndarray:
    """Inverse of :func:`pack_records`: (n, W) uint32 -> (n, 128) signed codes."""
    b = np.asarray(bits, np.int64)
    w64 = np.asarray(words).astype(np.uint64)
    u = np.zeros((w64.shape[0], len(b)), dtype=np.uint64)
    d2, d1 = record_entries(b)
    for i, (c, sh) in enumerate(d2):
        u[:, c] |= ((w64[:, i // 16] >> np.uint64(2 * (i % 16))) & np.uint64(3)) << np.uint64(sh)
    base = len(d2) // 16
    for j, (c, sh) in enumerate(d1):
        u[:, c] |= ((w64[:, base + j // 32] >> np.uint64(j % 32)) & np.uint64(1)) << np.uint64(sh)
    off = np.where(b > 0, 2 ** np.maximum(b - 1, 0), 0)
    return np.where(b[None, :] > 0, u.astype(np.int64) - off[None, :], 0)


QUARTER_POS = (0, 2, 1, 3)      # slot position of byte-quarter r inside a value slot block


def value_slot_of(token_in_tile: int, quarter: int) -> tuple:
    """Values are stored quad-interleaved: tokens 4Q..4Q+3 of a tile share the four slots
    4Q..4Q+3 of every record word; slot 4Q + QUARTER_POS[r] holds byte-quarter r (bits
    8r..8r+7) of the four tokens' words, token 4Q + i in byte i.  Returns (slot, byte)."""
    q, i = divmod(token_in_tile, 4)
    return 4 * q + QUARTER_POS[quarter], i


def cache_geometry(batch: int, n_kv_heads: int, max_tokens: int, n_words: int) -> dict:
    """Per-layer packed cache: uint32 words [batch][H_kv][2][n_tiles][W][128], then fp32 alpha
    [batch][H_kv][2][n_tiles*128].  Keys: token t of a sequence sits in tile t // 128, lane
    t % 128.  Values: slots as :func:`value_slot_of` says."""
    n_tiles = (max_tokens + TILE - 1) // TILE
    n_word_elems = batch * n_kv_heads * 2 * n_tiles * n_words * TILE
    n_alpha = batch * n_kv_heads * 2 * n_tiles * TILE
    return {"n_tiles": n_tiles, "words": n_word_elems, "alpha": n_alpha,
            "bytes": 4 * (n_word_elems + n_alpha)}


def cache_records(cache_u32: np.ndarray, batch: int, n_kv_heads: int, max_tokens: int,
                  n_words: int, b: int, head: int, kind: int, t0: int, n: int):
    """Read (records (n, W) uint32, alpha (n,) float32) of one stream back out of a cache image."""
    geo = cache_geometry(batch, n_kv_heads, max_tokens, n_words)
    nt = geo["n_tiles"]
    words = np.asarray(cache_u32[: geo["words"]]).reshape(batch, n_kv_heads, 2, nt, n_words, TILE)
    alpha = np.asarray(cache_u32[geo["words"]: geo["words"] + geo["alpha"]]).view(np.float32)
    alpha = alpha.reshape(batch, n_kv_heads, 2, nt * TILE)
    t = np.arange(t0, t0 + n)
    if kind == 0:
        rec = words[b, head, kind][t // TILE, :, t % TILE]        # (n, W)
    else:
        rec = np.zeros((n, n_words), dtype=np.uint64)
        for r in range(4):
            slots = np.array([value_slot_of(int(x), r)[0] for x in t % TILE], dtype=np.int64)
            byte = (t % TILE) % 4
            w = words[b, head, kind][t // TILE, :, slots].astype(np.uint64)      # (n, W)
            rec |= ((w >> (8 * byte[:, None]).astype(np.uint64)) & np.uint64(0xFF)) << np.uint64(8 * r)
        rec = rec.astype(np.uint32)
    return rec, alpha[b, head, kind, t0:t0 + n]


def cache_image(records_k, records_v, alpha_k, alpha_v, batch, n_kv_heads, max_tokens, n_words):
    """Build a whole-layer cache image (uint32) from per-stream records (for tests): records_x
    [batch][H_kv] -> (max_tokens, W) uint32 arrays; alpha_x [batch][H_kv] -> (max_tokens,)."""
    geo = cache_geometry(batch, n_kv_heads, max_tokens, n_words)
    nt = geo["n_tiles"]
    words = np.zeros((batch, n_kv_heads, 2, nt, n_words, TILE), np.uint32)
    alpha = np.zeros((batch, n_kv_heads, 2, nt * TILE), np.float32)
    for b in range(batch):
        for h in range(n_kv_heads):
            rk = records_k[b][h]
            for t in range(rk.shape[0]):
                words[b, h, 0, t // TILE, :, t % TILE] = rk[t]
            rv = records_v[b][h]
            for t in range(rv.shape[0]):
                for w in range(n_words):
                    x = int(rv[t, w])
                    for r in range(4):
                        slot, byte = value_slot_of(t % TILE, r)
                        cur = int(words[b, h, 1, t // TILE, w, slot])
                        cur = (cur & ~(0xFF << (8 * byte))) | (((x >> (8 * r)) & 0xFF) << (8 * byte))
                        words[b, h, 1, t // TILE, w, slot] = cur
            alpha[b, h, 0, :rk.shape[0]] = alpha_k[b][h]
            alpha[b, h, 1, :rv.shape[0]] = alpha_v[b][h]
    return np.concatenate([words.reshape(-1), alpha.reshape(-1).view(np.uint32)])


# ----------------------------------------------------------------------------
# Decode attention (Def. sdpa with one query row; Algorithm 1 inference lines)
# ----------------------------------------------------------------------------

def softmax(s: np.ndarray) -> np.ndarray:
    s = np.asarray(s, np.float64)
    e = np.exp(s - np.max(s))
    return e / np.sum(e)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, w_o: np.ndarray | None = None):
    """Single decode-step SDPA: s_i = q.k_i / sqrt(d_k), a = softmax(s), o = sum_i a_i v_i W_O
    (Def. sdpa, Eq. singleheadattoutput)."""
    q = np.asarray(q, np.float64)
    a = softmax(np.asarray(k, np.float64) @ q / math.sqrt(q.shape[-1]))
    o = a @ np.asarray(v, np.float64)
    return o if w_o is None else o @ np.asarray(w_o, np.float64)


def decode_attention(q_heads: np.ndarray, hk: np.ndarray, hv: np.ndarray, basis_k: np.ndarray,
                     basis_v: np.ndarray, group: int) -> np.ndarray:
    """Decode over coded coefficients of one sequence and layer (Alg. 1 reconstruct/attend lines).

    q_heads: (H_q, 128); hk, hv: (H_kv, n, 128) dequantized coefficients in storage order;
    basis_k, basis_v: (H_kv, 128, 128) reconstruction bases (K_hat = h_hat U^T).
    The keys are never rebuilt: q . (U h) = (U^T q) . h, and the value transform is applied
    once to the weighted sum.  Query head j reads kv-head j // group.
    """
    out = np.zeros((q_heads.shape[0], D))
    for j in range(q_heads.shape[0]):
        h = j // group
        qt = np.asarray(basis_k[h], np.float64).T @ np.asarray(q_heads[j], np.float64)
        a = softmax(np.asarray(hk[h], np.float64) @ qt / math.sqrt(D))
        out[j] = np.asarray(basis_v[h], np.float64) @ (a @ np.asarray(hv[h], np.float64))
    return out


# ----------------------------------------------------------------------------
# Head-group bases (Sec. 5 Step 1, remark on multi-head attention): the kv-heads of a group share
# one transform of width 128 G_h; every query head still attends with its own 128-dim block.
# ----------------------------------------------------------------------------

def embed_query(q: np.ndarray, block: int, n_blocks: int) -> np.ndarray:
    """A query head's vector placed at its kv-head's 128-dim block of the group's concatenated
    space (zeros elsewhere), so q . k_block = q_embedded . k_group."""
    q = np.asarray(q, np.float64)
    out = np.zeros(q.shape[:-1] + (D * n_blocks,))
    out[..., D * block:D * (block + 1)] = q
    return out


def plan_head_group(x_calib_heads: np.ndarray, avg_bits: float, b_max: int = 8, queries_by_head=None,
                    group: int = 1, weights: str = "aatc"):
    """Calibrate one head-group stream: the G_h kv-heads of the group (x_calib_heads: (G_h, N, 128),
    the same N calibration tokens) are concatenated into 128 G_h-dim vectors, which get one PCA
    basis, one weighted reverse water-filling over all 128 G_h channels with budget
    avg_bits * 128 G_h (Eq. waterfilling-keys over the group's channels) and one P99 scale per
    channel -- the steps of :func:`plan_stream` at the group's width.

    queries_by_head: for keys, the calibration queries of the group's query heads in kv-head
    order (G_h * group arrays of (T, 128)); query head i belongs to kv-head i // group, and its
    weight contribution uses the query embedded at that kv-head's block (the score it sees is
    q . k_block).  None for values (w = 1, W_O = I).  weights = 'var' gives w = 1 (var-only).
    """
    xh = np.asarray(x_calib_heads, np.float64)
    g_h = xh.shape[0]
    x = np.concatenate([xh[m] for m in range(g_h)], axis=1)           # (N, 128 G_h)
    width = D * g_h
    c = second_moment(x)
    lam, u = eigenbasis(c)
    if weights == "var" or queries_by_head is None:
        w = np.ones(width) if weights == "var" else value_weights(u.T)
    else:
        embedded = [embed_query(q, i // group, g_h) for i, q in enumerate(queries_by_head)]
        w = key_weights(u.T, embedded)
    gsc = w * lam
    order = np.argsort(-gsc, kind="stable")
    u, lam, w, gsc = u[:, order], lam[order], w[order], gsc[order]
    bits = greedy_allocation(gsc, int(round(avg_bits * width)), b_max)
    scales = channel_scales(u, x)
    return {"basis": u, "bits": bits, "scales": scales, "sigma2": lam, "weights": w, "g": gsc}


def decode_attention_head_group(q_heads: np.ndarray, hk: np.ndarray, hv: np.ndarray, basis_k: np.ndarray,
                                basis_v: np.ndarray, group: int) -> np.ndarray:
    """Decode over one head-group stream of one sequence (Alg. 1 reconstruct / attend lines at the
    group's width): q_heads (G_h * group, 128) are the group's query heads in kv-head order;
    hk, hv (n, 128 G_h) the dequantized group coefficients; basis_k, basis_v (128 G_h, 128 G_h)
    the group transforms (K_group_hat = h_hat U^T).  Query head i reads kv-head block m = i // group:
    s = (U_K^T q~) . h_hat / sqrt(128) with q~ the embedded query (the head dimension stays 128),
    a = softmax(s), out = (U_V (a h_hat^V)) restricted to block m."""
    hk = np.asarray(hk, np.float64)
    hv = np.asarray(hv, np.float64)
    g_h = hk.shape[1] // D
    out = np.zeros((q_heads.shape[0], D))
    for i in range(q_heads.shape[0]):
        m = i // group
        qt = np.asarray(basis_k, np.float64).T @ embed_query(q_heads[i], m, g_h)
        a = softmax(hk @ qt / math.sqrt(D))
        out[i] = (np.asarray(basis_v, np.float64) @ (a @ hv))[D * m:D * (m + 1)]
    return out


def prefill_attention(q_tokens: np.ndarray, positions: np.ndarray, hk: np.ndarray, hv: np.ndarray,
                      basis_k: np.ndarray, basis_v: np.ndarray, group: int) -> np.ndarray:
    """Causal attention of a chunk of new tokens over the coded cache of one sequence (Def. sdpa
    applied to every query row of the chunk; the cached coefficients stand in for K, V as in
    Alg. 1's reconstruct / attend lines).  q_tokens: (n_q, H_q, 128) queries at absolute
    positions `positions` (n_q,); hk, hv: (H_kv, n_ctx, 128) dequantized coefficients; query
    token at position p attends to cached tokens 0 .. p.  Returns (n_q, H_q, 128)."""
    out = np.zeros((q_tokens.shape[0], q_tokens.shape[1], D))
    for i, pos in enumerate(np.asarray(positions, np.int64)):
        out[i] = decode_attention(q_tokens[i], hk[:, :pos + 1], hv[:, :pos + 1], basis_k, basis_v, group)
    return out


def decode_attention_mixed(q_heads: np.ndarray, hk: np.ndarray, hv: np.ndarray, basis_k: np.ndarray,
                           basis_v: np.ndarray, group: int, k_full: np.ndarray, v_full: np.ndarray) -> np.ndarray:
    """Decode over coded tokens and uncompressed tokens in one softmax (the paper's inference
    policy keeps an attention sink and a recent window in full precision, Sec. 6 setup).

    hk, hv: (H_kv, n_coded, 128) dequantized coefficients; k_full, v_full: (H_kv, n_full, 128) in
    the original basis.  Scores: (U_K^T q) . h_hat / sqrt(128) for coded tokens, q . k / sqrt(128)
    for the others; a = softmax over both; out = U_V (sum_coded a h_hat^V) + sum_full a v.
    """
    out = np.zeros((q_heads.shape[0], D))
    for j in range(q_heads.shape[0]):
        h = j // group
        q = np.asarray(q_heads[j], np.float64)
        qt = np.asarray(basis_k[h], np.float64).T @ q
        s_c = np.asarray(hk[h], np.float64) @ qt / math.sqrt(D)
        s_f = np.asarray(k_full[h], np.float64) @ q / math.sqrt(D)
        a = softmax(np.concatenate([s_c, s_f]))
        n_c = s_c.shape[0]
        out[j] = (np.asarray(basis_v[h], np.float64) @ (a[:n_c] @ np.asarray(hv[h], np.float64))
                  + a[n_c:] @ np.asarray(v_full[h], np.float64))
    return out


def sink_window_counts(n_tokens: int, sink: int = 4, window: int = 128, step: int = 16):
    """Token accounting of the full-precision sink and recent window (Sec. 6 setup: first 4 tokens
    kept, a 128-token window moved in steps of 16).  Reading: the window fills up to
    window + step tokens; adding the token that makes it window + step flushes its oldest `step`
    tokens to the coded cache.  Returns (n_sink, n_coded, n_window) after n_tokens tokens; the
    coded tokens are positions [n_sink, n_sink + n_coded)."""
    n_sink = min(n_tokens, sink)
    rest = n_tokens - n_sink
    n_coded = step * max(0, (rest - window) // step)
    return n_sink, n_coded, rest - n_coded


# ----------------------------------------------------------------------------
# Theorem 1 (attention-output distortion decomposition)
# ----------------------------------------------------------------------------

def distortion_decomposition(q, k, v, var_k, var_v, w_o=None):
    """D_K and D_V of Theorem 1 for one decode step.

    D_K = sum_{i,c} a_i^2 ||v_i W_O - o||^2 q_c^2 E[dk_ic^2] and
    D_V = sum_{i,c} a_i^2 E[dv_ic^2] ||W_O,c||^2, where q_c is read as the c-th component of
    q / sqrt(d_k), the sensitivity of the score s_i to k_ic under Def. sdpa's scaling.
    """
    q = np.asarray(q, np.float64)
    k = np.asarray(k, np.float64)
    v = np.asarray(v, np.float64)
    d = q.shape[-1]
    wo = np.eye(v.shape[1]) if w_o is None else np.asarray(w_o, np.float64)
    a = softmax(k @ q / math.sqrt(d))
    vw = v @ wo
    o = a @ vw
    qe = q / math.sqrt(d)
    resid = np.sum((vw - o) ** 2, axis=1)
    dk = float(np.sum(a ** 2 * resid * (np.asarray(var_k) @ (qe ** 2))))
    dv = float(np.sum(a ** 2 * (np.asarray(var_v) @ np.sum(wo ** 2, axis=1))))
    return dk, dv
