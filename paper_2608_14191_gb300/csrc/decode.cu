// AATC decode attention over the packed cache, the dequantization test hook, and the
// uncompressed bf16 reference decode (Def. sdpa with one query row; Algorithm 1
// "Reconstruct", "softmax", "Output" lines, computed without rebuilding the keys).
//
// Split-K over the context (flash-decoding): one CTA per (split, kv-head, sequence) computes,
// for the G query heads of its GQA group,
//   phase 1  scores s_{g,t} = alpha^K_t * sum_c q'_{g,c} code^K_{t,c}   (thread = token),
//            with q' = (U_K^T q) * f^K * log2(e) / sqrt(128) folded once per CTA,
//   phase 2  split max m_g, p = 2^(s - m_g), l_g = sum p, P' = p * alpha^V_t,
//   phase 3  acc_{g,c} = sum_t P'_{g,t} code^V_{t,c}   (thread = 4 channels x 1/4 of the tokens),
// and writes (acc, m, l).  The combine kernel merges the splits by log-sum-exp, applies f^V and
// the one inverse value transform out = U_V o_hat.
#include <cuda_bf16.h>

#include <algorithm>
#include <mutex>

#include "aatc_internal.h"

namespace aatc {
namespace {

constexpr int kThreads = 128;
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_group 0;" ::: "memory"); }

// Block-wide max / sum of GP values per thread (128 threads).
template <int GP, bool kMax>
__device__ __forceinline__ void block_reduce(float (&v)[GP], float* scratch /* [4][GP] */) {
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float w = __shfl_xor_sync(0xffffffffu, v[g], o);
      v[g] = kMax ? fmaxf(v[g], w) : v[g] + w;
    }
  const int warp = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0)
#pragma unroll
    for (int g = 0; g < GP; ++g) scratch[warp * GP + g] = v[g];
  __syncthreads();
#pragma unroll
  for (int g = 0; g < GP; ++g) {
    float r = scratch[g];
#pragma unroll
    for (int w = 1; w < 4; ++w) r = kMax ? fmaxf(r, scratch[w * GP + g]) : r + scratch[w * GP + g];
    v[g] = r;
  }
  __syncthreads();
}

struct DecodeArgs {
  const uint32_t* words;   // cache word region (this layer)
  const float* alpha;      // cache alpha region
  const __nv_bfloat16* q;  // [batch][HQ][128]
  float* ws;               // [batch][HQ][n_splits][130]
  const float* u32;        // plan: [S][128 dim][128 ch]
  const float* f;          // plan: [S][128]
  const int* ext;          // plan: [S][128]
  const int* nret;         // plan: [S]
  int layer, n_kv, n_q, group, n_ctx, n_tiles, n_words, n_splits, split_len;
};

// Shared-memory plan of the split kernel (floats unless noted).
template <int GP>
struct SplitSmem {
  static constexpr int kQt = 0;                                 // [128][GP] folded query
  static constexpr int kQf = kQt + D * GP;                      // [GP][128] query (fp32)
  static constexpr int kCg = kQf + GP * D;                      // [GP] offset corrections
  static constexpr int kRed = kCg + 8;                          // [4][8] reductions
  static constexpr int kExtK = kRed + 32;                       // int [128] (offset | b << 16)
  static constexpr int kAlpha = kExtK + D;                      // [2][128] alpha of the staged tile
  static constexpr int kScores = kAlpha + 2 * TILE;             // [split_len][GP]
  // followed by the word tiles: [2][(W + 2) * 132] u32, then acc scratch [4][GP][128]
};

template <int GP>
__global__ void __launch_bounds__(kThreads)
    aatc_decode_split_kernel(const DecodeArgs a) {
  extern __shared__ __align__(16) float sm[];
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x;
  const int G = a.group;
  const int sk = (a.layer * a.n_kv + head) * 2;                 // key stream; value = sk + 1
  const int RK = a.nret[sk], RV = a.nret[sk + 1];
  using L = SplitSmem<GP>;
  float* qt = sm + L::kQt;
  float* qf = sm + L::kQf;
  float* cg = sm + L::kCg;
  float* red = sm + L::kRed;
  int* extk = reinterpret_cast<int*>(sm + L::kExtK);
  float* al = sm + L::kAlpha;
  float* sc = sm + L::kScores;
  const int stride = 132;                                       // padded word-plane stride (u32)
  uint32_t* wt = reinterpret_cast<uint32_t*>(sc + a.split_len * GP);   // [2][(W+2)*132]
  const int wt_elems = (a.n_words + 2) * stride;
  float* accs = reinterpret_cast<float*>(wt + 2 * wt_elems);    // [4][GP][128]

  const int t_begin = split * a.split_len;
  const int t_end = min(a.n_ctx, t_begin + a.split_len);
  const int n_tiles_split = (t_end - t_begin + TILE - 1) / TILE;
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;
  const size_t bk = (static_cast<size_t>(b) * a.n_kv + head) * 2;   // cache stream index of K
  const uint32_t* kwords = a.words + bk * stream_words;
  const uint32_t* vwords = a.words + (bk + 1) * stream_words;
  const float* kalpha = a.alpha + bk * a.n_tiles * TILE;
  const float* valpha = a.alpha + (bk + 1) * a.n_tiles * TILE;

  // ---- prologue: folded query q'_{g,c} = (U_K^T q_g)_c f_c log2e / sqrt(128)
  for (int i = tid; i < GP * D; i += kThreads) {
    const int g = i / D, d = i % D;
    qf[i] = g < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + g) * D + d]) : 0.0f;
  }
  extk[tid] = a.ext[sk * D + tid];
  __syncthreads();
  {
    const int c = tid;
    float accq[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) accq[g] = 0.0f;
    const float* uk = a.u32 + static_cast<size_t>(sk) * D * D;
    for (int d = 0; d < D; ++d) {
      const float u = uk[d * D + c];
#pragma unroll
      for (int g = 0; g < GP; ++g) accq[g] = fmaf(u, qf[g * D + d], accq[g]);
    }
    const float fk = a.f[sk * D + c] * (kLog2e * 0.08838834764831845f);   // 1/sqrt(128)
    const int bits = extk[c] >> 16;
    const float off = bits > 0 ? static_cast<float>(1 << (bits - 1)) : 0.0f;
    float corr[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float v = c < RK ? accq[g] * fk : 0.0f;
      qt[c * GP + g] = v;
      corr[g] = v * off;
    }
    block_reduce<GP, false>(corr, red);
    if (tid < GP) cg[tid] = corr[tid];
  }
  __syncthreads();

  // ---- phase 1: scores, thread = token
  auto stage_tile = [&](const uint32_t* src_words, const float* src_alpha, int tile, int buf) {
    uint32_t* dst = wt + buf * wt_elems;
    const uint32_t* src = src_words + static_cast<size_t>(tile) * a.n_words * TILE;
    const int chunks = a.n_words * (TILE / 4);
    for (int i = tid; i < chunks; i += kThreads) {
      const int w = i / (TILE / 4), q4 = i % (TILE / 4);
      cp_async16(dst + w * stride + q4 * 4, src + w * TILE + q4 * 4);
    }
    if (tid < TILE / 4) cp_async16(al + buf * TILE + tid * 4, src_alpha + tile * TILE + tid * 4);
    cp_async_commit();
  };
  // zero the two guard planes once (read past the record by the sliding window)
  for (int i = tid; i < 2 * stride; i += kThreads) {
    wt[a.n_words * stride + i] = 0u;
    wt[wt_elems + a.n_words * stride + i] = 0u;
  }
  const int tile0 = t_begin / TILE;
  stage_tile(kwords, kalpha, tile0, 0);
  float mloc[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) mloc[g] = -INFINITY;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage_tile(kwords, kalpha, tile0 + ti + 1, buf ^ 1);
    const uint32_t* w = wt + buf * wt_elems;
    float s[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) s[g] = 0.0f;
    uint32_t lo = w[tid], hi = w[stride + tid];
    int cw = 0;
    for (int c = 0; c < RK; ++c) {
      const int e = extk[c];
      const int o = e & 0xFFFF;
      const int nb = e >> 16;
      if ((o >> 5) != cw) {                     // uniform: advance the two-word window
        cw = o >> 5;
        lo = hi;
        hi = w[(cw + 1) * stride + tid];
      }
      const uint32_t x = __funnelshift_r(lo, hi, o & 31);
      const uint32_t u = (x & ((1u << nb) - 1u)) | 0x4B000000u;
      const float cf = __uint_as_float(u) - 8388608.0f;
      if constexpr (GP == 4) {
        const float4 qv = *reinterpret_cast<const float4*>(qt + c * 4);
        s[0] = fmaf(qv.x, cf, s[0]);
        s[1] = fmaf(qv.y, cf, s[1]);
        s[2] = fmaf(qv.z, cf, s[2]);
        s[3] = fmaf(qv.w, cf, s[3]);
      } else {
#pragma unroll
        for (int g4 = 0; g4 < GP; g4 += 4) {
          const float4 qv = *reinterpret_cast<const float4*>(qt + c * GP + g4);
          s[g4] = fmaf(qv.x, cf, s[g4]);
          s[g4 + 1] = fmaf(qv.y, cf, s[g4 + 1]);
          s[g4 + 2] = fmaf(qv.z, cf, s[g4 + 2]);
          s[g4 + 3] = fmaf(qv.w, cf, s[g4 + 3]);
        }
      }
    }
    const int t = (tile0 + ti) * TILE + tid;
    const float ak = al[buf * TILE + tid];
    const bool valid = t < t_end;
    float* out = sc + (ti * TILE + tid) * GP;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float v = valid ? ak * (s[g] - cg[g]) : -INFINITY;
      out[g] = v;
      mloc[g] = fmaxf(mloc[g], v);
    }
  }
  cp_async_wait_all();
  __syncthreads();

  // ---- phase 2: split max, probabilities (scaled by alpha^V), split sum
  block_reduce<GP, true>(mloc, red);
  stage_tile(vwords, valpha, tile0, 0);
  float lsum[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) lsum[g] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    float* p = sc + (ti * TILE + tid) * GP;
    const int t = (tile0 + ti) * TILE + tid;
    const float av = t < t_end ? valpha[t] : 0.0f;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float e = exp2f(p[g] - mloc[g]);     // exp2(-inf) = 0 for padding tokens
      lsum[g] += e;
      p[g] = e * av;
    }
  }
  block_reduce<GP, false>(lsum, red);

  // ---- phase 3: value accumulation, thread = (4 channels, token quarter)
  const int cgp = tid & 31, tq = tid >> 5;
  const int c0 = cgp * 4;
  int ws_ = 0, sh0 = 0, rel[4], msk[4];
  float kof[4];
  {
    const int* ev = a.ext + (sk + 1) * D;
    const int o0 = ev[c0] & 0xFFFF;
    ws_ = o0 >> 5;
    sh0 = o0 & 31;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int c = c0 + i;
      const int e = ev[c];
      const int nb = c < RV ? (e >> 16) : 0;
      rel[i] = (e & 0xFFFF) - o0;
      msk[i] = nb > 0 ? ((1 << nb) - 1) : 0;
      kof[i] = 8388608.0f + (nb > 0 ? static_cast<float>(1 << (nb - 1)) : 0.0f);
    }
  }
  float acc[GP][4];
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[g][i] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage_tile(vwords, valpha, tile0 + ti + 1, buf ^ 1);
    const uint32_t* w = wt + buf * wt_elems;
    const int tend = min(TILE, t_end - (tile0 + ti) * TILE);
    for (int tt = tq; tt < tend; tt += 4) {
      const uint32_t x = __funnelshift_r(w[ws_ * stride + tt], w[(ws_ + 1) * stride + tt], sh0);
      const float* p = sc + (ti * TILE + tt) * GP;
      float cf[4];
#pragma unroll
      for (int i = 0; i < 4; ++i)
        cf[i] = __uint_as_float(((x >> rel[i]) & static_cast<uint32_t>(msk[i])) | 0x4B000000u) - kof[i];
#pragma unroll
      for (int g4 = 0; g4 < GP; g4 += 4) {
        const float4 pv = *reinterpret_cast<const float4*>(p + g4);
        const float pg[4] = {pv.x, pv.y, pv.z, pv.w};
#pragma unroll
        for (int gg = 0; gg < 4; ++gg)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[g4 + gg][i] = fmaf(pg[gg], cf[i], acc[g4 + gg][i]);
      }
    }
  }
  cp_async_wait_all();
  __syncthreads();
  // reduce the four token quarters
#pragma unroll
  for (int g = 0; g < GP; ++g)
    *reinterpret_cast<float4*>(accs + (tq * GP + g) * D + c0) = make_float4(acc[g][0], acc[g][1], acc[g][2], acc[g][3]);
  __syncthreads();
  for (int g = 0; g < G; ++g) {
    const float v = accs[(0 * GP + g) * D + tid] + accs[(1 * GP + g) * D + tid] + accs[(2 * GP + g) * D + tid] +
                    accs[(3 * GP + g) * D + tid];
    float* dst = a.ws + ((static_cast<size_t>(b) * a.n_q + head * G + g) * a.n_splits + split) * (D + 2);
    dst[tid] = v;
    if (tid == 0) {
      dst[D] = mloc[g];
      dst[D + 1] = lsum[g];
    }
  }
}

// Merge the splits of one (sequence, query head) by log-sum-exp, scale by f^V and apply U_V.
// With u32 == nullptr the transform is the identity (bf16 reference path).
__global__ void __launch_bounds__(kThreads)
    aatc_decode_combine_kernel(const float* ws, int n_splits, int n_q, int group, const float* u32, const float* f,
                               int layer, int n_kv, float* out) {
  __shared__ float ohat[D];
  __shared__ float red[8];
  const int j = blockIdx.x, b = blockIdx.y, tid = threadIdx.x;
  const int head = j / group;
  const float* src = ws + (static_cast<size_t>(b) * n_q + j) * n_splits * (D + 2);
  float m = -INFINITY;
  for (int s = tid; s < n_splits; s += kThreads) m = fmaxf(m, src[s * (D + 2) + D]);
  float mv[1] = {m};
  block_reduce<1, true>(mv, red);
  m = mv[0];
  float l = 0.0f;
  for (int s = tid; s < n_splits; s += kThreads) l += src[s * (D + 2) + D + 1] * exp2f(src[s * (D + 2) + D] - m);
  float lv[1] = {l};
  block_reduce<1, false>(lv, red);
  const float inv_l = 1.0f / lv[0];
  float acc = 0.0f;
  for (int s = 0; s < n_splits; ++s) acc += src[s * (D + 2) + tid] * exp2f(src[s * (D + 2) + D] - m);
  const int sv = (layer * n_kv + head) * 2 + 1;
  const float fv = u32 ? f[sv * D + tid] : 1.0f;
  ohat[tid] = acc * inv_l * fv;
  __syncthreads();
  float o;
  if (u32) {
    const float* uv = u32 + static_cast<size_t>(sv) * D * D + tid * D;
    o = 0.0f;
    for (int c = 0; c < D; ++c) o = fmaf(uv[c], ohat[c], o);
  } else {
    o = ohat[tid];
  }
  out[(static_cast<size_t>(b) * n_q + j) * D + tid] = o;
}

// Dequantization hook: thread per (sequence, token, stream) of the requested range.
__global__ void aatc_dequant_kernel(const uint32_t* words, const float* alpha, const int* ext, const float* f,
                                    int layer, int n_kv, int batch, int t0, int n, int n_tiles, int n_words,
                                    float* out) {
  const long idx = static_cast<long>(blockIdx.x) * blockDim.x + threadIdx.x;
  const long total = static_cast<long>(batch) * n * n_kv * 2;
  if (idx >= total) return;
  const int kind = static_cast<int>(idx % 2);
  const int head = static_cast<int>((idx / 2) % n_kv);
  const int i = static_cast<int>((idx / (2 * n_kv)) % n);
  const int b = static_cast<int>(idx / (2L * n_kv * n));
  const int t = t0 + i;
  const size_t cs = (static_cast<size_t>(b) * n_kv + head) * 2 + kind;
  const uint32_t* rec = words + cs * n_tiles * n_words * TILE + static_cast<size_t>(t / TILE) * n_words * TILE + t % TILE;
  const float at = alpha[cs * n_tiles * TILE + t];
  const int s = (layer * n_kv + head) * 2 + kind;
  float* o = out + idx * D;
  for (int c = 0; c < D; ++c) {
    const int e = ext[s * D + c];
    const int off = e & 0xFFFF, nb = e >> 16;
    float v = 0.0f;
    if (nb > 0) {
      const int w = off >> 5, sh = off & 31;
      const uint32_t lo = rec[static_cast<size_t>(w) * TILE];
      const uint32_t hi = (sh + nb > 32) ? rec[static_cast<size_t>(w + 1) * TILE] : 0u;
      const uint32_t u = __funnelshift_r(lo, hi, sh) & ((1u << nb) - 1u);
      const int code = static_cast<int>(u) - (1 << (nb - 1));
      const float delta = __fmul_rn(at, f[s * D + c]);
      v = __fmul_rn(static_cast<float>(code), delta);
    }
    o[c] = v;
  }
}

// ---------------------------------------------------------------- bf16 reference decode
struct Bf16Args {
  const __nv_bfloat16* k;  // [batch][max_tokens][n_kv][128]
  const __nv_bfloat16* v;
  const __nv_bfloat16* q;  // [batch][n_q][128]
  float* ws;
  int n_kv, n_q, group, n_ctx, max_tokens, n_splits, split_len;
};

__device__ __forceinline__ void bf16x8_to_f32(const uint4 r, float* o) {
  const uint32_t w[4] = {r.x, r.y, r.z, r.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    o[2 * i] = __uint_as_float(w[i] << 16);
    o[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

template <int GP>
__global__ void __launch_bounds__(kThreads)
    aatc_bf16_split_kernel(const Bf16Args a) {
  extern __shared__ __align__(16) float sm[];
  const int split = blockIdx.x, head = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int G = a.group;
  constexpr int kRow = D + 8;                              // padded bf16 row (272 B)
  float* qs = sm;                                          // [128][GP]
  float* red = qs + D * GP;                                // [32]
  float* sc = red + 32;                                    // [split_len][GP]
  __nv_bfloat16* kt = reinterpret_cast<__nv_bfloat16*>(sc + a.split_len * GP);   // [2][128][kRow]
  float* accs = reinterpret_cast<float*>(kt + 2 * TILE * kRow);                  // [4][GP][128]
  const int t_begin = split * a.split_len;
  const int t_end = min(a.n_ctx, t_begin + a.split_len);
  const int n_tiles_split = (t_end - t_begin + TILE - 1) / TILE;
  const float scale = kLog2e * 0.08838834764831845f;
  for (int i = tid; i < GP * D; i += kThreads) {
    const int g = i / D, d = i % D;
    qs[d * GP + g] =
        g < G ? __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q + head * G + g) * D + d]) * scale : 0.0f;
  }
  auto stage = [&](const __nv_bfloat16* base, int tile, int buf) {
    __nv_bfloat16* dst = kt + buf * TILE * kRow;
    for (int i = tid; i < TILE * 16; i += kThreads) {
      const int r = i >> 4, ch = i & 15;
      int t = tile * TILE + r;
      t = min(t, a.n_ctx - 1);                             // clamp padding rows to a valid token
      cp_async16(dst + r * kRow + ch * 8, base + ((static_cast<size_t>(b) * a.max_tokens + t) * a.n_kv + head) * D + ch * 8);
    }
    cp_async_commit();
  };
  const int tile0 = t_begin / TILE;
  stage(a.k, tile0, 0);
  __syncthreads();
  float mloc[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) mloc[g] = -INFINITY;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage(a.k, tile0 + ti + 1, buf ^ 1);
    const __nv_bfloat16* row = kt + buf * TILE * kRow + tid * kRow;
    float s[GP];
#pragma unroll
    for (int g = 0; g < GP; ++g) s[g] = 0.0f;
    for (int d0 = 0; d0 < D; d0 += 8) {
      float kv[8];
      bf16x8_to_f32(*reinterpret_cast<const uint4*>(row + d0), kv);
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int g4 = 0; g4 < GP; g4 += 4) {
          const float4 qv = *reinterpret_cast<const float4*>(qs + (d0 + i) * GP + g4);
          s[g4] = fmaf(qv.x, kv[i], s[g4]);
          s[g4 + 1] = fmaf(qv.y, kv[i], s[g4 + 1]);
          s[g4 + 2] = fmaf(qv.z, kv[i], s[g4 + 2]);
          s[g4 + 3] = fmaf(qv.w, kv[i], s[g4 + 3]);
        }
    }
    const int t = (tile0 + ti) * TILE + tid;
    float* out = sc + (ti * TILE + tid) * GP;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float v = t < t_end ? s[g] : -INFINITY;
      out[g] = v;
      mloc[g] = fmaxf(mloc[g], v);
    }
  }
  cp_async_wait_all();
  __syncthreads();
  block_reduce<GP, true>(mloc, red);
  stage(a.v, tile0, 0);
  float lsum[GP];
#pragma unroll
  for (int g = 0; g < GP; ++g) lsum[g] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    float* p = sc + (ti * TILE + tid) * GP;
#pragma unroll
    for (int g = 0; g < GP; ++g) {
      const float e = exp2f(p[g] - mloc[g]);
      lsum[g] += e;
      p[g] = e;
    }
  }
  block_reduce<GP, false>(lsum, red);
  const int dg = tid & 31, tq = tid >> 5;
  float acc[GP][4];
#pragma unroll
  for (int g = 0; g < GP; ++g)
#pragma unroll
    for (int i = 0; i < 4; ++i) acc[g][i] = 0.0f;
  for (int ti = 0; ti < n_tiles_split; ++ti) {
    const int buf = ti & 1;
    cp_async_wait_all();
    __syncthreads();
    if (ti + 1 < n_tiles_split) stage(a.v, tile0 + ti + 1, buf ^ 1);
    const int tend = min(TILE, t_end - (tile0 + ti) * TILE);
    for (int tt = tq; tt < tend; tt += 4) {
      const uint2 r = *reinterpret_cast<const uint2*>(kt + buf * TILE * kRow + tt * kRow + dg * 4);
      const float vv[4] = {__uint_as_float(r.x << 16), __uint_as_float(r.x & 0xFFFF0000u),
                           __uint_as_float(r.y << 16), __uint_as_float(r.y & 0xFFFF0000u)};
      const float* p = sc + (ti * TILE + tt) * GP;
#pragma unroll
      for (int g4 = 0; g4 < GP; g4 += 4) {
        const float4 pv = *reinterpret_cast<const float4*>(p + g4);
        const float pg[4] = {pv.x, pv.y, pv.z, pv.w};
#pragma unroll
        for (int gg = 0; gg < 4; ++gg)
#pragma unroll
          for (int i = 0; i < 4; ++i) acc[g4 + gg][i] = fmaf(pg[gg], vv[i], acc[g4 + gg][i]);
      }
    }
  }
  cp_async_wait_all();
  __syncthreads();
#pragma unroll
  for (int g = 0; g < GP; ++g)
    *reinterpret_cast<float4*>(accs + (tq * GP + g) * D + dg * 4) = make_float4(acc[g][0], acc[g][1], acc[g][2], acc[g][3]);
  __syncthreads();
  for (int g = 0; g < G; ++g) {
    const float v = accs[(0 * GP + g) * D + tid] + accs[(1 * GP + g) * D + tid] + accs[(2 * GP + g) * D + tid] +
                    accs[(3 * GP + g) * D + tid];
    float* dst = a.ws + ((static_cast<size_t>(b) * a.n_q + head * G + g) * a.n_splits + split) * (D + 2);
    dst[tid] = v;
    if (tid == 0) {
      dst[D] = mloc[g];
      dst[D + 1] = lsum[g];
    }
  }
}

template <int GP>
size_t split_smem_bytes(int split_len, int n_words) {
  using L = SplitSmem<GP>;
  return 4 * (static_cast<size_t>(L::kScores) + static_cast<size_t>(split_len) * GP + 2 * (n_words + 2) * 132 +
              4 * GP * D);
}

template <int GP>
cudaError_t launch_split(const DecodeArgs& a, int batch, int n_kv, cudaStream_t st) {
  const size_t smem = split_smem_bytes<GP>(a.split_len, a.n_words);
  static size_t smem_set = 0;                                  // raise the opt-in limit only when needed
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(aatc_decode_split_kernel<GP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  aatc_decode_split_kernel<GP><<<dim3(a.n_splits, n_kv, batch), kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

template <int GP>
cudaError_t launch_bf16_split(const Bf16Args& a, int batch, cudaStream_t st) {
  const size_t smem = 4 * (static_cast<size_t>(D) * GP + 32 + static_cast<size_t>(a.split_len) * GP + 4 * GP * D) +
                      2 * static_cast<size_t>(TILE) * (D + 8) * 2;
  static size_t smem_set = 0;
  if (smem > smem_set) {
    cudaError_t e = cudaFuncSetAttribute(aatc_bf16_split_kernel<GP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    smem_set = smem;
  }
  aatc_bf16_split_kernel<GP><<<dim3(a.n_splits, a.n_kv, batch), kThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                          int max_tokens, float* out, void* ws, const DecodeSplit& sp, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  DecodeArgs a;
  a.words = static_cast<const uint32_t*>(cache);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.ws = static_cast<float*>(ws);
  a.u32 = plan.dev.u32;
  a.f = plan.dev.f;
  a.ext = plan.dev.ext;
  a.nret = plan.dev.nret;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.n_q = plan.dims.n_q_heads;
  a.group = a.n_q / a.n_kv;
  a.n_ctx = n_ctx;
  a.n_tiles = g.n_tiles;
  a.n_words = plan.n_words;
  a.n_splits = sp.n_splits;
  a.split_len = sp.split_len;
  cudaError_t e = a.group <= 4 ? launch_split<4>(a, batch, a.n_kv, st) : launch_split<8>(a, batch, a.n_kv, st);
  if (e != cudaSuccess) return e;
  aatc_decode_combine_kernel<<<dim3(a.n_q, batch), kThreads, 0, st>>>(a.ws, a.n_splits, a.n_q, a.group, plan.dev.u32,
                                                                     plan.dev.f, layer, a.n_kv, out);
  return cudaGetLastError();
}

cudaError_t launch_dequant(const Plan& plan, int layer, const void* cache, int batch, int t0, int n, int max_tokens,
                           float* out, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  const long total = static_cast<long>(batch) * n * plan.dims.n_kv_heads * 2;
  const int threads = 128;
  const long blocks = (total + threads - 1) / threads;
  aatc_dequant_kernel<<<static_cast<unsigned>(blocks), threads, 0, st>>>(
      static_cast<const uint32_t*>(cache), reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems),
      plan.dev.ext, plan.dev.f, layer, plan.dims.n_kv_heads, batch, t0, n, g.n_tiles, plan.n_words, out);
  return cudaGetLastError();
}

cudaError_t launch_bf16_decode(const void* K, const void* V, const void* q, int batch, int n_ctx, int max_tokens,
                               int n_kv, int n_q, float* out, void* ws, const DecodeSplit& sp, cudaStream_t st) {
  Bf16Args a;
  a.k = static_cast<const __nv_bfloat16*>(K);
  a.v = static_cast<const __nv_bfloat16*>(V);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.ws = static_cast<float*>(ws);
  a.n_kv = n_kv;
  a.n_q = n_q;
  a.group = n_q / n_kv;
  a.n_ctx = n_ctx;
  a.max_tokens = max_tokens;
  a.n_splits = sp.n_splits;
  a.split_len = sp.split_len;
  cudaError_t e = a.group <= 4 ? launch_bf16_split<4>(a, batch, st) : launch_bf16_split<8>(a, batch, st);
  if (e != cudaSuccess) return e;
  aatc_decode_combine_kernel<<<dim3(n_q, batch), kThreads, 0, st>>>(a.ws, a.n_splits, n_q, a.group, nullptr, nullptr, 0,
                                                                     n_kv, out);
  return cudaGetLastError();
}

}  // namespace aatc

// ------------------------------------------------------------------ decode without a workspace
// For callers that cannot allocate device memory at call time (see aatc_decode_attention_noalloc
// in aatc.h): the split partials live in one fixed array of this file, reserved on every device
// that loads the library.  Host code must not use the array's name as an address; the device
// address is looked up once per device with cudaGetSymbolAddress.
namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[AATC_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_noalloc_mutex;
void* g_noalloc_address[kMaxDevices] = {};

}  // namespace

extern "C" aatc_status_t aatc_decode_attention_noalloc(aatc_plan_t p, int32_t layer, const void* q,
                                                       const void* cache, int32_t batch, int32_t n_ctx,
                                                       int32_t max_tokens, float* out, void* stream) {
  using namespace aatc;
  Plan* plan = plan_from_handle(p);
  if (!plan || !q || !cache || !out || layer < 0 || layer >= plan->dims.n_layers || batch < 1 || n_ctx < 1 ||
      max_tokens < 1)
    return AATC_ERR_INVALID_ARG;
  if (n_ctx > max_tokens) return AATC_ERR_CAPACITY;
  if (plan->dims.n_q_heads / plan->dims.n_kv_heads > MAX_GROUP) return AATC_ERR_UNSUPPORTED;
  if ((reinterpret_cast<uintptr_t>(cache) & 15u) != 0) return AATC_ERR_INVALID_ARG;
  const DecodeSplit sp = decode_split(batch, plan->dims.n_kv_heads, n_ctx, plan->num_sms);
  if (decode_workspace(batch, plan->dims.n_q_heads, sp) > AATC_NOALLOC_SCRATCH_BYTES) return AATC_ERR_WORKSPACE;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return status_from_cuda(e);
  if (dev < 0 || dev >= kMaxDevices) return AATC_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mutex);
    if (!g_noalloc_address[dev]) {
      e = cudaGetSymbolAddress(&g_noalloc_address[dev], g_noalloc_scratch);
      if (e != cudaSuccess) {
        g_noalloc_address[dev] = nullptr;
        return status_from_cuda(e);
      }
    }
    scratch = g_noalloc_address[dev];
  }
  return status_from_cuda(launch_decode(*plan, layer, q, cache, batch, n_ctx, max_tokens, out, scratch, sp,
                                        static_cast<cudaStream_t>(stream)));
}
