// Prefill attention over the packed cache: a chunk of new query tokens attends causally to the
// cached tokens (Def. sdpa for every query row; Algorithm 1's reconstruct / attend lines, computed
// in the transformed space as the decode does: q . (U h) = (U^T q) . h).
//
// Two launches per call:
//   codes    per (128-token tile, kv-head x K|V, sequence): the packed records -> the signed codes
//            code_c = u_c - 2^(b_c - 1) as f16 (exact: |code| <= 128), [b][h][K|V][n_ctx_pad][128];
//   attn     per (64 query rows, kv-head, sequence), rows = (query token, head of the GQA group):
//            q' = (U_K^T q) f^K log2(e) / sqrt(128) as f16 hi/lo (CUDA cores, fp32), then per
//            64-token tile S = alpha^K (q'_hi + q'_lo) . code^K (mma.sync m16n8k16), causal mask,
//            online softmax, P' = 2^(S - m) alpha^V (f16) and O += P' code^V, finally
//            out = U_V (f^V O / l) (CUDA cores, fp32).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "aatc_internal.h"

namespace aatc {
namespace {

constexpr int kPThreads = 128;      // 4 warps x 16 query rows
constexpr int kPRows = 64;
constexpr int kPKV = 64;            // cached tokens per tile
constexpr int kPStride = D + 8;     // f16 row stride of the code tiles (272 B: ldmatrix rows in distinct banks)
constexpr float kPLog2e = 1.4426950408889634f;
constexpr float kPOpMax = 16384.0f; // q' rows scaled so the largest |value| is 2^14

struct PrefillArgs {
  const uint32_t* words;     // cache word region (this layer)
  const float* alpha;        // cache alpha region
  const __nv_bfloat16* q;    // [batch][n_q][H_q][128]
  float* out;                // [batch][n_q][H_q][128]
  __half* codes;             // workspace [batch][n_kv][2][n_ctx_pad][128]
  const float* u32;          // plan: [S][128 dim][128 ch]
  const float* u32t;         // plan: [S][128 ch][128 dim]
  const float* f;            // plan: [S][128]
  const ChanEnc* enc;        // plan: [S][128] (offsets 2^(b-1))
  const StreamLayout* lay;   // plan: [S]
  const short* entry;        // plan: [S][n_entries]
  const short* chan_ent;     // plan: [S][128][8]
  int layer, n_kv, n_q_heads, group, q_start, n_q, n_ctx, n_ctx_pad, n_tiles, n_words, n_entries;
};

__global__ void __launch_bounds__(TILE) aatc_prefill_codes_kernel(const PrefillArgs a) {
  __shared__ uint32_t rec[32][TILE];           // record words of the tile's tokens (W <= 32)
  const int tile = blockIdx.x, hk = blockIdx.y, b = blockIdx.z, t = threadIdx.x;
  const int head = hk >> 1, kind = hk & 1;
  const size_t cs = (static_cast<size_t>(b) * a.n_kv + head) * 2 + kind;
  const int tok = tile * TILE + t;
  __half* dst = a.codes + (cs * a.n_ctx_pad + tok) * D;
  if (tok >= a.n_ctx) {                        // padding rows of the last tile: zero codes
    if (tok < a.n_ctx_pad)
      for (int c = 0; c < D; c += 8) *reinterpret_cast<uint4*>(dst + c) = make_uint4(0u, 0u, 0u, 0u);
    return;
  }
  const int s = (a.layer * a.n_kv + head) * 2 + kind;
  const StreamLayout ly = a.lay[s];
  const int nw = ly.n2 / 16 + (ly.n1 + 31) / 32;
  const uint32_t* tw = a.words + (cs * a.n_tiles + tile) * static_cast<size_t>(a.n_words) * TILE;
  for (int w = 0; w < nw; ++w) {
    const uint32_t* ww = tw + static_cast<size_t>(w) * TILE;
    uint32_t x;
    if (kind == 0) {
      x = ww[t];
    } else {                                   // quad-interleaved: quarter r in slot 4Q + (0, 2, 1, 3)[r]
      const int q4 = 4 * (t >> 2), sh = 8 * (t & 3);
      x = ((ww[q4] >> sh) & 0xFFu) | (((ww[q4 + 2] >> sh) & 0xFFu) << 8) | (((ww[q4 + 1] >> sh) & 0xFFu) << 16) |
          (((ww[q4 + 3] >> sh) & 0xFFu) << 24);
    }
    rec[w][t] = x;                             // each thread reads back only its own column
  }
  const short* ce = a.chan_ent + static_cast<size_t>(s) * D * 8;
  const short* ent = a.entry + static_cast<size_t>(s) * a.n_entries;
  for (int c = 0; c < D; c += 2) {
    float v2[2];
#pragma unroll
    for (int i = 0; i < 2; ++i) {
      const int cc = c + i;
      uint32_t u = 0;
      for (int k = 0; k < 8; ++k) {
        const int e = ce[cc * 8 + k];
        if (e < 0) break;
        uint32_t v;
        if (e < ly.n2) {
          v = (rec[e >> 4][t] >> (2 * (e & 15))) & 3u;
        } else {
          const int e1 = e - ly.n2;
          v = (rec[ly.n2 / 16 + (e1 >> 5)][t] >> (e1 & 31)) & 1u;
        }
        u |= v << ((ent[e] >> 8) & 7);
      }
      v2[i] = static_cast<float>(u) - a.enc[s * D + cc].off;   // dropped channels: u = off = 0
    }
    *reinterpret_cast<__half2*>(dst + c) = __floats2half2_rn(v2[0], v2[1]);
  }
}

__device__ __forceinline__ void mma16816(float (&c)[4], const uint32_t (&a)[4], uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}
__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ float ex2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
__device__ __forceinline__ uint32_t pack_h2(float lo, float hi) {
  const __half2 h = __floats2half2_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

struct PrefillSmem {
  __half kc[2][kPKV][kPStride];
  __half vc[2][kPKV][kPStride];
  float ak[2][kPKV], av[2][kPKV];
  float qs[kPRows][D];          // q (fp32), then q', then o_hat
};

__global__ void __launch_bounds__(kPThreads) aatc_prefill_attn_kernel(const PrefillArgs a) {
  extern __shared__ __align__(16) unsigned char psm[];
  PrefillSmem& sm = *reinterpret_cast<PrefillSmem*>(psm);
  const int rb = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, g = lane >> 2, t = lane & 3;
  const int G = a.group, n_rows = a.n_q * G;
  const int sk = (a.layer * a.n_kv + head) * 2, sv = sk + 1;
  const size_t csk = (static_cast<size_t>(b) * a.n_kv + head) * 2, csv = csk + 1;
  // rows of this CTA: R = 64 rb + r -> query token R / G, head head * G + R % G
  auto row_pos = [&](int r) { return a.q_start + (rb * kPRows + r) / G; };
  const int r_last = min(n_rows - 1, rb * kPRows + kPRows - 1) - rb * kPRows;
  const int kv_end = min(a.n_ctx, row_pos(r_last) + 1);       // tokens [0, kv_end) can be attended
  const int n_kv_tiles = (kv_end + kPKV - 1) / kPKV;

  auto load_tile = [&](int jt, int buf) {
    const __half* kg = a.codes + (csk * a.n_ctx_pad + static_cast<size_t>(jt) * kPKV) * D;
    const __half* vg = a.codes + (csv * a.n_ctx_pad + static_cast<size_t>(jt) * kPKV) * D;
    for (int i = tid; i < kPKV * (D / 8); i += kPThreads) {
      const int r = i >> 4, c8 = (i & 15) * 8;
      cp_async16(&sm.kc[buf][r][c8], kg + r * D + c8);
      cp_async16(&sm.vc[buf][r][c8], vg + r * D + c8);
    }
    if (tid < kPKV) {
      const int tok = jt * kPKV + tid;
      sm.ak[buf][tid] = a.alpha[csk * a.n_tiles * TILE + tok];
      sm.av[buf][tid] = a.alpha[csv * a.n_tiles * TILE + tok];
    }
    asm volatile("cp.async.commit_group;" ::: "memory");
  };
  if (n_kv_tiles > 0) load_tile(0, 0);

  // ---- q' rows: q (bf16 -> fp32) into shared memory, then (U_K^T q) f^K log2(e) / sqrt(128)
  for (int i = tid; i < kPRows * D; i += kPThreads) {
    const int r = i >> 7, d = i & (D - 1);
    const int R = rb * kPRows + r;
    float v = 0.0f;
    if (R < n_rows) {
      const int qi = R / G, qh = head * G + R % G;
      v = __bfloat162float(a.q[((static_cast<size_t>(b) * a.n_q + qi) * a.n_q_heads + qh) * D + d]);
    }
    sm.qs[r][d] = v;
  }
  __syncthreads();
  float rs[2];                                  // score scale of rows g, g + 8 of this warp
  {
    // warp = 16 rows, lane = channels 4 lane .. 4 lane + 3
    float acc[16][4];
#pragma unroll
    for (int r = 0; r < 16; ++r)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[r][j] = 0.0f;
    const float* uk = a.u32 + static_cast<size_t>(sk) * D * D + 4 * lane;
    for (int d = 0; d < D; ++d) {
      const float4 u4 = *reinterpret_cast<const float4*>(uk + d * D);
#pragma unroll
      for (int r = 0; r < 16; ++r) {
        const float qv = sm.qs[16 * warp + r][d];
        acc[r][0] = fmaf(qv, u4.x, acc[r][0]);
        acc[r][1] = fmaf(qv, u4.y, acc[r][1]);
        acc[r][2] = fmaf(qv, u4.z, acc[r][2]);
        acc[r][3] = fmaf(qv, u4.w, acc[r][3]);
      }
    }
    const float4 f4 = *reinterpret_cast<const float4*>(a.f + sk * D + 4 * lane);
    const float sc = kPLog2e * 0.08838834764831845f;
    float mx[16];
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      acc[r][0] *= f4.x * sc;
      acc[r][1] *= f4.y * sc;
      acc[r][2] *= f4.z * sc;
      acc[r][3] *= f4.w * sc;
      float m = fmaxf(fmaxf(fabsf(acc[r][0]), fabsf(acc[r][1])), fmaxf(fabsf(acc[r][2]), fabsf(acc[r][3])));
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
      mx[r] = m;
    }
    __syncwarp();
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      const float inv = mx[r] > 0.0f ? kPOpMax / mx[r] : 0.0f;
      *reinterpret_cast<float4*>(&sm.qs[16 * warp + r][4 * lane]) =
          make_float4(acc[r][0] * inv, acc[r][1] * inv, acc[r][2] * inv, acc[r][3] * inv);
    }
    rs[0] = rs[1] = 0.0f;
    // mx[] is indexed by g (lane-dependent): pick without local memory
#pragma unroll
    for (int r = 0; r < 8; ++r)
      if (r == g) {
        rs[0] = mx[r] / kPOpMax;
        rs[1] = mx[r + 8] / kPOpMax;
      }
  }
  __syncwarp();
  // A fragments of q' (rows g, g + 8 of this warp), hi and lo
  uint32_t qh[8][4], ql[8][4];
#pragma unroll
  for (int ks = 0; ks < 8; ++ks) {
    const float* r0 = sm.qs[16 * warp + g];
    const float* r1 = sm.qs[16 * warp + g + 8];
    const int k0 = 16 * ks + 2 * t, k1 = k0 + 8;
    const float v[8] = {r0[k0], r0[k0 + 1], r1[k0], r1[k0 + 1], r0[k1], r0[k1 + 1], r1[k1], r1[k1 + 1]};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const __half2 h = __floats2half2_rn(v[2 * j], v[2 * j + 1]);
      const float2 hf = __half22float2(h);
      qh[ks][j] = *reinterpret_cast<const uint32_t*>(&h);
      ql[ks][j] = pack_h2(v[2 * j] - hf.x, v[2 * j + 1] - hf.y);
    }
  }
  const int pos0 = row_pos(16 * warp + g), pos1 = row_pos(16 * warp + g + 8);

  // ---- online softmax over the cached tokens
  float o[16][4];
#pragma unroll
  for (int n = 0; n < 16; ++n)
#pragma unroll
    for (int j = 0; j < 4; ++j) o[n][j] = 0.0f;
  float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.0f, l1 = 0.0f;
  for (int jt = 0; jt < n_kv_tiles; ++jt) {
    const int buf = jt & 1;
    if (jt + 1 < n_kv_tiles) {
      load_tile(jt + 1, buf ^ 1);
      asm volatile("cp.async.wait_group 1;" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;" ::: "memory");
    }
    __syncthreads();
    float s[8][4];
#pragma unroll
    for (int n = 0; n < 8; ++n)
#pragma unroll
      for (int j = 0; j < 4; ++j) s[n][j] = 0.0f;
#pragma unroll
    for (int np = 0; np < 4; ++np)
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        // matrices: tokens 16np + (0..7 | 8..15) x channels 16ks + (0..7 | 8..15)
        const int mi = lane >> 3;
        uint32_t bb[4];
        ldsm_x4(bb, &sm.kc[buf][16 * np + (mi >> 1) * 8 + (lane & 7)][16 * ks + (mi & 1) * 8]);
        mma16816(s[2 * np], qh[ks], bb[0], bb[1]);
        mma16816(s[2 * np], ql[ks], bb[0], bb[1]);
        mma16816(s[2 * np + 1], qh[ks], bb[2], bb[3]);
        mma16816(s[2 * np + 1], ql[ks], bb[2], bb[3]);
      }
    // scores: rows g (c0, c1) and g + 8 (c2, c3), tokens 64 jt + 8n + 2t + {0, 1}
    float mt0 = m0, mt1 = m1;
#pragma unroll
    for (int n = 0; n < 8; ++n)
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int tl = 8 * n + 2 * t + (j & 1), tok = jt * kPKV + tl;
        const bool row1 = j >= 2;
        const bool ok = tok <= (row1 ? pos1 : pos0) && tok < a.n_ctx;
        const float v = ok ? s[n][j] * (row1 ? rs[1] : rs[0]) * sm.ak[buf][tl] : -INFINITY;
        s[n][j] = v;
        if (row1) mt1 = fmaxf(mt1, v); else mt0 = fmaxf(mt0, v);
      }
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      mt0 = fmaxf(mt0, __shfl_xor_sync(0xffffffffu, mt0, off));
      mt1 = fmaxf(mt1, __shfl_xor_sync(0xffffffffu, mt1, off));
    }
    const float c0 = mt0 == -INFINITY ? 1.0f : ex2(m0 - mt0), c1 = mt1 == -INFINITY ? 1.0f : ex2(m1 - mt1);
    m0 = mt0;
    m1 = mt1;
    l0 *= c0;
    l1 *= c1;
#pragma unroll
    for (int n = 0; n < 16; ++n) {
      o[n][0] *= c0;
      o[n][1] *= c0;
      o[n][2] *= c1;
      o[n][3] *= c1;
    }
    uint32_t pa[4][4];                          // P' A fragments, k16-step = 16 tokens
#pragma unroll
    for (int n = 0; n < 8; ++n) {
      float p[4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        const int tl = 8 * n + 2 * t + (j & 1);
        const float mm = j >= 2 ? m1 : m0;
        const float e = s[n][j] == -INFINITY ? 0.0f : ex2(s[n][j] - mm);
        if (j >= 2) l1 += e; else l0 += e;
        p[j] = e * sm.av[buf][tl];
        if (s[n][j] == -INFINITY) p[j] = 0.0f;
      }
      pa[n >> 1][(n & 1) * 2 + 0] = pack_h2(p[0], p[1]);     // row g, tokens 2t, 2t+1 (+8 for odd n)
      pa[n >> 1][(n & 1) * 2 + 1] = pack_h2(p[2], p[3]);     // row g + 8
    }
#pragma unroll
    for (int ks2 = 0; ks2 < 4; ++ks2) {
      // A: a0 = (row g, k 2t..), a1 = (row g+8, k 2t..), a2 = (row g, k 2t+8..), a3 = (row g+8, k 2t+8..)
      const uint32_t af[4] = {pa[ks2][0], pa[ks2][1], pa[ks2][2], pa[ks2][3]};
#pragma unroll
      for (int cp = 0; cp < 8; ++cp) {
        // matrices: tokens 16ks2 + (0..7 | 8..15) x channels 16cp + (0..7 | 8..15), transposed
        const int mi = lane >> 3;
        uint32_t bb[4];
        ldsm_x4_t(bb, &sm.vc[buf][16 * ks2 + (mi & 1) * 8 + (lane & 7)][16 * cp + (mi >> 1) * 8]);
        mma16816(o[2 * cp], af, bb[0], bb[1]);
        mma16816(o[2 * cp + 1], af, bb[2], bb[3]);
      }
    }
    __syncthreads();                            // buffer `buf` is refilled by the next iteration
  }
  // ---- o_hat = f^V O / l, then out = U_V o_hat
#pragma unroll
  for (int off = 1; off < 4; off <<= 1) {
    l0 += __shfl_xor_sync(0xffffffffu, l0, off);
    l1 += __shfl_xor_sync(0xffffffffu, l1, off);
  }
  const float il0 = l0 > 0.0f ? 1.0f / l0 : 0.0f, il1 = l1 > 0.0f ? 1.0f / l1 : 0.0f;
  __syncwarp();
#pragma unroll
  for (int n = 0; n < 16; ++n) {
    const int c = 8 * n + 2 * t;
    const float f0 = a.f[sv * D + c], f1 = a.f[sv * D + c + 1];
    sm.qs[16 * warp + g][c] = o[n][0] * il0 * f0;
    sm.qs[16 * warp + g][c + 1] = o[n][1] * il0 * f1;
    sm.qs[16 * warp + g + 8][c] = o[n][2] * il1 * f0;
    sm.qs[16 * warp + g + 8][c + 1] = o[n][3] * il1 * f1;
  }
  __syncwarp();
  {
    float acc[16][4];
#pragma unroll
    for (int r = 0; r < 16; ++r)
#pragma unroll
      for (int j = 0; j < 4; ++j) acc[r][j] = 0.0f;
    const float* ut = a.u32t + static_cast<size_t>(sv) * D * D + 4 * lane;   // [ch][dim]
    for (int c = 0; c < D; ++c) {
      const float4 u4 = *reinterpret_cast<const float4*>(ut + c * D);
#pragma unroll
      for (int r = 0; r < 16; ++r) {
        const float ov = sm.qs[16 * warp + r][c];
        acc[r][0] = fmaf(ov, u4.x, acc[r][0]);
        acc[r][1] = fmaf(ov, u4.y, acc[r][1]);
        acc[r][2] = fmaf(ov, u4.z, acc[r][2]);
        acc[r][3] = fmaf(ov, u4.w, acc[r][3]);
      }
    }
#pragma unroll
    for (int r = 0; r < 16; ++r) {
      const int R = rb * kPRows + 16 * warp + r;
      if (R < n_rows) {
        const int qi = R / G, qh2 = head * G + R % G;
        *reinterpret_cast<float4*>(a.out + ((static_cast<size_t>(b) * a.n_q + qi) * a.n_q_heads + qh2) * D + 4 * lane) =
            make_float4(acc[r][0], acc[r][1], acc[r][2], acc[r][3]);
      }
    }
  }
}

}  // namespace

size_t prefill_workspace(int batch, int n_kv, int n_ctx) {
  const size_t pad = (static_cast<size_t>(n_ctx) + TILE - 1) / TILE * TILE;
  return static_cast<size_t>(batch) * n_kv * 2 * pad * D * sizeof(__half);
}

cudaError_t launch_prefill(const Plan& plan, int layer, const void* q, int q_start, int n_q, const void* cache,
                           int batch, int n_ctx, int max_tokens, float* out, void* ws, cudaStream_t st) {
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  PrefillArgs a;
  a.words = static_cast<const uint32_t*>(cache);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.out = out;
  a.codes = static_cast<__half*>(ws);
  a.u32 = plan.dev.u32;
  a.u32t = plan.dev.u32t;
  a.f = plan.dev.f;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.entry = plan.dev.entry;
  a.chan_ent = plan.dev.chan_ent;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.n_q_heads = plan.dims.n_q_heads;
  a.group = a.n_q_heads / a.n_kv;
  a.q_start = q_start;
  a.n_q = n_q;
  a.n_ctx = n_ctx;
  a.n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  a.n_tiles = g.n_tiles;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  if (plan.n_words > 32) return cudaErrorNotSupported;
  aatc_prefill_codes_kernel<<<dim3(a.n_ctx_pad / TILE, a.n_kv * 2, batch), TILE, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  static bool attr_done = false;
  const size_t smem = sizeof(PrefillSmem);
  if (!attr_done) {
    e = cudaFuncSetAttribute(aatc_prefill_attn_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr_done = true;
  }
  const int n_rows = n_q * a.group;
  aatc_prefill_attn_kernel<<<dim3((n_rows + kPRows - 1) / kPRows, a.n_kv, batch), kPThreads, smem, st>>>(a);
  return cudaGetLastError();
}

}  // namespace aatc
