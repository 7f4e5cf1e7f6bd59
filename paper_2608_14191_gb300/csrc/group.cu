// Decode attention over head-group streams (Sec. 5 Step 1, remark on multi-head attention: the
// g_h kv-heads of a group share one transform; Def. sdpa per query head, Algorithm 1's
// reconstruct / attend / output lines in the transformed space).
//
// A group stream of n = 128 g_h channels is stored as g_h slice streams in the per-kv-head slots
// (slice s = storage channels s, s + g_h, ...), one alpha per token.  Query head j of the group
// (kv-head block m = j / group) sees the embedded query q~ (q at block m, zeros elsewhere):
//   score_t = (U_K^T q~) . h_hat_t / sqrt(128) = alpha_t sum_c q'_c f_c code_tc,
//   out     = rows of block m of U_V applied to sum_t p_t h_hat^V_t.
// Four launches per call:
//   codes  every slice's signed codes as f16 (exact for widths <= 8), rebuilt in closed form from
//          the record layout's run bounds
//   query  per (query head, group, sequence): q'' = (U_K^T q~) f log2(e) / sqrt(128) over the n
//          slice-major channels (thread = channel)
//   attn   per (split, group, sequence), 8 warps: per 128-token tile the key codes of every slice
//          (S = q''_hi . code + q''_lo . code, mma.sync m16n8k16 f16, rows = the group's <= 16
//          query heads, one accumulator over all n channels), online softmax with the exponent of
//          alpha^V folded into the running maximum (so P' = 2^(s - m) alpha^V stays below 2), then
//          O_s += P' . code^V for every slice s; row operands from shared memory by ldmatrix
//   merge  per (query head, group, sequence): log-sum-exp over the splits, o_hat = f^V O / l, and
//          out = U_V[block m rows] o_hat
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "aatc_internal.h"
#include "ptx.cuh"

namespace aatc {
namespace {

constexpr float kGLog2e = 1.4426950408889634f;
constexpr int kGAThreads = 256;                  // 8 warps
constexpr int kGRing = 4;                        // code chunks in flight
constexpr int kGRowHalves = D + 8;               // padded shared-memory row (272 bytes)

struct GroupDecodeArgs {
  const __half* codes;       // codes workspace [b][n_kv][K|V][n_ctx_pad][128]
  const float* alpha;        // cache alpha region [b][n_kv][K|V][n_tiles * 128]
  const __nv_bfloat16* q;    // [b][H_q][128]
  const float* uk;           // plan: U_K of every (layer, group), [n dim][n channel]
  const float* uvt;          // plan: U_V^T, [n channel][n dim]
  const float* f;            // plan: [slot][128] f_c
  float* qf;                 // workspace: folded queries [b][n_groups][nq][n]
  float* part;               // workspace: split partials [b][n_groups][nq][n_splits][n + 4]
  float* out;                // [b][H_q][128]
  int layer, n_kv, gh, n_groups, group, nq, n, n_q_heads, n_ctx, n_ctx_pad, n_tiles, n_splits;
};

__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(static_cast<uint32_t>(__cvta_generic_to_shared(dst))),
               "l"(src)
               : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}
// Four 8x8 b16 matrices; lane l gives the address of row l % 8 of matrix l / 8.
__device__ __forceinline__ void ldmatrix_x4(uint32_t (&r)[4], const void* p) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
               : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
               : "r"(static_cast<uint32_t>(__cvta_generic_to_shared(p))));
}
__device__ __forceinline__ void mma16816(float (&c)[4], const uint4& a, uint32_t b0, uint32_t b1) {
  asm volatile(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
      "{%0, %1, %2, %3};"
      : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
      : "r"(a.x), "r"(a.y), "r"(a.z), "r"(a.w), "r"(b0), "r"(b1));
}
__device__ __forceinline__ float fexp2(float x) {
  float r;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}
// f16 hi / lo parts of x and y, packed as (x, y) pairs
__device__ __forceinline__ void split2(float x, float y, uint32_t& hi, uint32_t& lo) {
  const __half2 h = __floats2half2_rn(x, y);
  const float2 hf = __half22float2(h);
  const __half2 l = __floats2half2_rn(x - hf.x, y - hf.y);
  hi = *reinterpret_cast<const uint32_t*>(&h);
  lo = *reinterpret_cast<const uint32_t*>(&l);
}

// Signed codes of every slot's records as f16 (exact for widths <= 8), in the prefill codes
// layout ([b][slot][K|V][n_ctx_pad][128]; value tiles transposed to [channel][token]).  Thread =
// token of one 128-token tile of one slot and kind.  Each stored value is rebuilt in closed form
// from the stream's run bounds (no entry tables): digit k of channel c (c < l2all[k]) is D2 entry
// sum_{k' < k} l2[k'] + c when c < l2[k], else the moved pair at D1 bit n_odd + 2 (moved before
// it); the top bit of a width 2k + 1 channel is D1 bit (odd channels of wider widths) + (c -
// l2all[k]).  Widths are non-increasing in storage order, which makes every run a prefix.
__global__ void __launch_bounds__(TILE) aatc_group_codes_kernel(const uint32_t* words, const StreamLayout* lays,
                                                                __half* codes, int layer, int n_kv, int n_ctx,
                                                                int n_ctx_pad, int n_tiles, int n_words) {
  __shared__ uint32_t rec[32][TILE];
  const int tile = blockIdx.x, hk = blockIdx.y, b = blockIdx.z, t = threadIdx.x;
  const int head = hk >> 1, kind = hk & 1;
  const size_t cs = (static_cast<size_t>(b) * n_kv + head) * 2 + kind;
  const int tok = tile * TILE + t;
  __half* krow = codes + (cs * n_ctx_pad + tok) * D;
  __half* vcol = codes + cs * n_ctx_pad * D + static_cast<size_t>(tile) * TILE * D + t;
  const __half zero = __float2half_rn(0.0f);
  if (tok >= n_ctx) {                              // padding tokens of the last tile: zero codes
    if (tok < n_ctx_pad) {
      if (kind == 1) {
        for (int c = 0; c < D; ++c) vcol[c * TILE] = zero;
      } else {
        for (int c = 0; c < D; c += 8) *reinterpret_cast<uint4*>(krow + c) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    return;
  }
  const StreamLayout ly = lays[(layer * n_kv + head) * 2 + kind];
  const int nw = ly.n2 / 16 + (ly.n1 + 31) / 32;
  const uint32_t* tw = words + (cs * n_tiles + tile) * static_cast<size_t>(n_words) * TILE;
  for (int w = 0; w < nw; ++w) {
    const uint32_t* ww = tw + static_cast<size_t>(w) * TILE;
    uint32_t x;
    if (kind == 0) {
      x = ww[t];
    } else {                                       // quad-interleaved: quarter r in slot 4Q + (0, 2, 1, 3)[r]
      const int q4 = 4 * (t >> 2), sh = 8 * (t & 3);
      x = ((ww[q4] >> sh) & 0xFFu) | (((ww[q4 + 2] >> sh) & 0xFFu) << 8) | (((ww[q4 + 1] >> sh) & 0xFFu) << 16) |
          (((ww[q4 + 3] >> sh) & 0xFFu) << 24);
    }
    rec[w][t] = x;                                 // each thread reads back only its own column
  }
  int e0[8], mo[8], od[8];
  int n_odd = 0;
  {
    int e = 0, m = 0;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      e0[k] = e;
      mo[k] = m;
      e += ly.l2[k];
      m += ly.l2all[k] - ly.l2[k];
    }
#pragma unroll
    for (int k = 7; k >= 0; --k) {
      od[k] = n_odd;
      n_odd += ly.lodd[k] - ly.l2all[k];
    }
  }
  const int d1w = ly.n2 / 16;
  auto d1bit = [&](int p) -> uint32_t { return (rec[d1w + (p >> 5)][t] >> (p & 31)) & 1u; };
  for (int c0 = 0; c0 < D; c0 += 8) {
    float v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int c = c0 + i;
      uint32_t u = 0;
      int nb = 0;
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        if (c >= ly.lodd[k]) break;                // lodd is non-increasing in k
        if (c < ly.l2all[k]) {
          uint32_t dg;
          if (c < ly.l2[k]) {
            const int e = e0[k] + c;
            dg = (rec[e >> 4][t] >> (2 * (e & 15))) & 3u;
          } else {
            const int p = n_odd + 2 * (mo[k] + c - ly.l2[k]);
            dg = d1bit(p) | (d1bit(p + 1) << 1);
          }
          u |= dg << (2 * k);
          nb = 2 * k + 2;
        } else {
          u |= d1bit(od[k] + c - ly.l2all[k]) << (2 * k);
          nb = 2 * k + 1;
        }
      }
      v[i] = nb > 0 ? static_cast<float>(static_cast<int>(u) - (1 << (nb - 1))) : 0.0f;
    }
    if (kind == 1) {
#pragma unroll
      for (int i = 0; i < 8; ++i) vcol[(c0 + i) * TILE] = __float2half_rn(v[i]);
    } else {
      uint4 q;
      q.x = *reinterpret_cast<const uint32_t*>(&(const __half2&)__floats2half2_rn(v[0], v[1]));
      q.y = *reinterpret_cast<const uint32_t*>(&(const __half2&)__floats2half2_rn(v[2], v[3]));
      q.z = *reinterpret_cast<const uint32_t*>(&(const __half2&)__floats2half2_rn(v[4], v[5]));
      q.w = *reinterpret_cast<const uint32_t*>(&(const __half2&)__floats2half2_rn(v[6], v[7]));
      *reinterpret_cast<uint4*>(krow + c0) = q;
    }
  }
}

// q'' of one query head over the group's n channels (thread = slice-major channel j' = 128 s + c).
__global__ void aatc_group_query_kernel(const GroupDecodeArgs a) {
  __shared__ float qv[D];
  const int i = blockIdx.x, g = blockIdx.y, b = blockIdx.z, j = threadIdx.x;
  const int m = i / a.group, hq = g * a.nq + i;
  if (j < D) qv[j] = __bfloat162float(a.q[(static_cast<size_t>(b) * a.n_q_heads + hq) * D + j]);
  __syncthreads();
  const float* u = a.uk + (static_cast<size_t>(a.layer) * a.n_groups + g) * a.n * a.n + static_cast<size_t>(m) * D * a.n;
  float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
  for (int d = 0; d < D; d += 16) {                // 16 loads in flight per thread
    float x[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) x[k] = u[static_cast<size_t>(d + k) * a.n + j];
#pragma unroll
    for (int k = 0; k < 16; ++k) acc[k & 3] = fmaf(x[k], qv[d + k], acc[k & 3]);
  }
  const int s = j / D, c = j % D;
  const int slot = (a.layer * a.n_kv + g * a.gh + s) * 2;
  a.qf[((static_cast<size_t>(b) * a.n_groups + g) * a.nq + i) * a.n + j] =
      ((acc[0] + acc[1]) + (acc[2] + acc[3])) * a.f[slot * D + c] * (kGLog2e * 0.08838834764831845f);
}

template <int GH>
struct GroupAttnSmem {
  static constexpr int N = D * GH, NKS = N / 16;
  uint4 qfrag[NKS][32][2];                        // score A fragments (hi, lo) per k-step and lane
  uint4 pfrag[TILE / 16][32][2];                  // P' A fragments (hi, lo) of the current tile
  alignas(128) __half ring[kGRing][TILE][kGRowHalves];
  float redm[8][16], reds[8][16];
  float qinv[16], mrow[16], lrow[16], rscale[16];
};

template <int GH>
__global__ void __launch_bounds__(kGAThreads, 1) aatc_group_attn_kernel(const GroupDecodeArgs a) {
  constexpr int N = D * GH, NKS = N / 16, NCH = 2 * GH;
  extern __shared__ __align__(128) unsigned char smb[];
  auto& sm = *reinterpret_cast<GroupAttnSmem<GH>*>(smb);
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, gq = lane >> 2, t = lane & 3;
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE;
  const int tile_lo = static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const size_t slot0 = static_cast<size_t>(b) * a.n_kv + static_cast<size_t>(g) * GH;   // cache slot of slice 0
  const float* kalpha = a.alpha + (slot0 * 2) * a.n_tiles * TILE;
  const float* valpha = a.alpha + (slot0 * 2 + 1) * a.n_tiles * TILE;
  const float* qf = a.qf + (static_cast<size_t>(b) * a.n_groups + g) * a.nq * N;

  // ---- score A fragments: rows = queries (>= nq zero), scaled by a power of two so the largest
  // |q''| of a row is below 2^14, split into f16 hi / lo
  if (tid < 16) {
    float mx = 0.0f;
    if (tid < a.nq)
      for (int j = 0; j < N; ++j) mx = fmaxf(mx, fabsf(qf[tid * N + j]));
    int ex = 0;
    if (mx > 0.0f) frexpf(mx, &ex);               // mx < 2^ex
    sm.qinv[tid] = ldexpf(1.0f, ex - 14);          // the row was scaled by 2^(14 - ex)
    sm.mrow[tid] = -INFINITY;
    sm.lrow[tid] = 0.0f;
  }
  __syncthreads();
  for (int idx = tid; idx < NKS * 32; idx += kGAThreads) {
    const int ks = idx >> 5, ln = idx & 31, r0 = ln >> 2, c0 = ks * 16 + 2 * (ln & 3);
    float v[8];
    const int rows[4] = {r0, r0 + 8, r0, r0 + 8};
    const int cols[4] = {c0, c0, c0 + 8, c0 + 8};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int r = rows[k];
      const float sc = r < a.nq ? 1.0f / sm.qinv[r] : 0.0f;
      v[2 * k] = r < a.nq ? qf[r * N + cols[k]] * sc : 0.0f;
      v[2 * k + 1] = r < a.nq ? qf[r * N + cols[k] + 1] * sc : 0.0f;
    }
    uint4 hi, lo;
    split2(v[0], v[1], hi.x, lo.x);
    split2(v[2], v[3], hi.y, lo.y);
    split2(v[4], v[5], hi.z, lo.z);
    split2(v[6], v[7], hi.w, lo.w);
    sm.qfrag[ks][ln][0] = hi;
    sm.qfrag[ks][ln][1] = lo;
  }

  // ---- code chunks: per tile the key codes of slices 0 .. GH-1, then their value codes
  const int n_chunks = (tile_hi - tile_lo) * NCH;
  auto issue = [&](int u) {
    if (u < n_chunks) {
      const int tile = tile_lo + u / NCH, c = u % NCH, s = c % GH, kind = c / GH;
      const __half* src = a.codes + ((slot0 + s) * 2 + kind) * static_cast<size_t>(a.n_ctx_pad) * D +
                          static_cast<size_t>(tile) * TILE * D;
      __half* dst = &sm.ring[u % kGRing][0][0];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int p = tid + kGAThreads * k, row = p >> 4, col = (p & 15) * 8;
        cp_async16(dst + row * kGRowHalves + col, src + row * D + col);
      }
    }
    cp_async_commit();
  };
  for (int u = 0; u < kGRing - 1; ++u) issue(u);

  float sacc[2][4];
  float oacc[GH][2][4];
#pragma unroll
  for (int s = 0; s < GH; ++s)
#pragma unroll
    for (int nt = 0; nt < 2; ++nt)
#pragma unroll
      for (int r = 0; r < 4; ++r) oacc[s][nt][r] = 0.0f;
  const int tw = 16 * warp;                       // score pass: this warp's tokens of the tile
  const int cw = 16 * warp;                       // value pass: this warp's channels of each slice
  // ldmatrix row addresses: matrix l / 8 = (rows +8 if l >= 16, columns +8 if l & 8)
  const int lrow = (lane & 7) + ((lane & 16) ? 8 : 0), lcol = (lane & 8) ? 8 : 0;

  for (int u = 0; u < n_chunks; ++u) {
    issue(u + kGRing - 1);
    cp_async_wait<kGRing - 1>();
    __syncthreads();
    const int tile = tile_lo + u / NCH, c = u % NCH, s = c % GH;
    const __half* ch = &sm.ring[u % kGRing][0][0];
    if (c < GH) {
      // ---- scores of this warp's 16 tokens over slice s
      if (s == 0)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int r = 0; r < 4; ++r) sacc[nt][r] = 0.0f;
#pragma unroll
      for (int ks = 0; ks < 8; ++ks) {
        uint32_t bm[4];
        ldmatrix_x4(bm, ch + (tw + lrow) * kGRowHalves + ks * 16 + lcol);
        const uint4 ah = sm.qfrag[s * 8 + ks][lane][0], al = sm.qfrag[s * 8 + ks][lane][1];
        mma16816(sacc[0], ah, bm[0], bm[1]);
        mma16816(sacc[0], al, bm[0], bm[1]);
        mma16816(sacc[1], ah, bm[2], bm[3]);
        mma16816(sacc[1], al, bm[2], bm[3]);
      }
      if (c == GH - 1) {
        // ---- online softmax of the tile.  Lane (gq, t) holds rows gq, gq + 8 and tokens
        // tw + 8 nt + 2t + {0, 1}; e = s + floor(log2 alpha^V) keeps P' = 2^(e - m) mant(alpha^V) < 2.
        float e[2][4], mant[2][4], lav[2][4];
        float mx0 = -INFINITY, mx1 = -INFINITY;
        const float qi0 = sm.qinv[gq], qi1 = sm.qinv[gq + 8];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            const int tok = tile * TILE + tw + 8 * nt + 2 * t + (r & 1);
            const int row = r < 2 ? gq : gq + 8;
            const bool ok = tok < a.n_ctx && row < a.nq;
            float ev = -INFINITY, mv = 0.0f, lv = 0.0f;
            if (ok) {
              const float ak = kalpha[tok], avv = valpha[tok];
              const float sv = sacc[nt][r] * (r < 2 ? qi0 : qi1) * ak;
              int ex = 0;
              const float fr = frexpf(avv, &ex);        // avv = fr 2^ex, fr in [0.5, 1)
              lv = avv > 0.0f ? static_cast<float>(max(ex - 1, -64)) : -64.0f;
              mv = avv > 0.0f ? fr * 2.0f : 0.0f;
              if (avv > 0.0f && ex - 1 < -64) mv = avv * 18446744073709551616.0f;   // alpha^V / 2^-64
              ev = sv + lv;
            }
            e[nt][r] = ev;
            mant[nt][r] = mv;
            lav[nt][r] = lv;
            if (r < 2) mx0 = fmaxf(mx0, ev);
            else mx1 = fmaxf(mx1, ev);
          }
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
        mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
        mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
        if (t == 0) {
          sm.redm[warp][gq] = mx0;
          sm.redm[warp][gq + 8] = mx1;
        }
        __syncthreads();
        if (tid < 16) {
          float mt = -INFINITY;
#pragma unroll
          for (int w = 0; w < 8; ++w) mt = fmaxf(mt, sm.redm[w][tid]);
          const float mo = sm.mrow[tid], mn = fmaxf(mo, mt);
          sm.rscale[tid] = mo == -INFINITY ? 0.0f : fexp2(mo - mn);
          sm.mrow[tid] = mn;
        }
        __syncthreads();
        const float m0 = sm.mrow[gq], m1 = sm.mrow[gq + 8];
        float ls0 = 0.0f, ls1 = 0.0f;
        float p[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            const float mm = r < 2 ? m0 : m1;
            const float x = e[nt][r] == -INFINITY ? 0.0f : fexp2(e[nt][r] - mm);   // 2^(e - m) <= 1
            p[nt][r] = x * mant[nt][r];                                           // P' = 2^(s - m) alpha^V
            const float l = e[nt][r] == -INFINITY ? 0.0f : x * exp2f(-lav[nt][r]);  // 2^(s - m)
            if (r < 2) ls0 += l;
            else ls1 += l;
          }
        uint4 ph, pl;
        split2(p[0][0], p[0][1], ph.x, pl.x);   // row gq,     tokens 2t, 2t + 1
        split2(p[0][2], p[0][3], ph.y, pl.y);   // row gq + 8, tokens 2t, 2t + 1
        split2(p[1][0], p[1][1], ph.z, pl.z);   // row gq,     tokens 2t + 8, 2t + 9
        split2(p[1][2], p[1][3], ph.w, pl.w);   // row gq + 8, tokens 2t + 8, 2t + 9
        sm.pfrag[warp][lane][0] = ph;
        sm.pfrag[warp][lane][1] = pl;
        ls0 += __shfl_xor_sync(0xffffffffu, ls0, 1);
        ls0 += __shfl_xor_sync(0xffffffffu, ls0, 2);
        ls1 += __shfl_xor_sync(0xffffffffu, ls1, 1);
        ls1 += __shfl_xor_sync(0xffffffffu, ls1, 2);
        if (t == 0) {
          sm.reds[warp][gq] = ls0;
          sm.reds[warp][gq + 8] = ls1;
        }
        const float r0 = sm.rscale[gq], r1 = sm.rscale[gq + 8];
#pragma unroll
        for (int s2 = 0; s2 < GH; ++s2)
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) {
            oacc[s2][nt][0] *= r0;
            oacc[s2][nt][1] *= r0;
            oacc[s2][nt][2] *= r1;
            oacc[s2][nt][3] *= r1;
          }
        __syncthreads();
        if (tid < 16) {
          float lt = 0.0f;
#pragma unroll
          for (int w = 0; w < 8; ++w) lt += sm.reds[w][tid];
          sm.lrow[tid] = sm.lrow[tid] * sm.rscale[tid] + lt;
        }
      }
    } else {
      // ---- O_s += P' . code^V: this warp's 16 channels of slice s, K = the tile's 128 tokens
#pragma unroll
      for (int kt = 0; kt < TILE / 16; ++kt) {
        uint32_t bm[4];
        ldmatrix_x4(bm, ch + (cw + lrow) * kGRowHalves + kt * 16 + lcol);
        const uint4 ah = sm.pfrag[kt][lane][0], al = sm.pfrag[kt][lane][1];
#pragma unroll
        for (int s2 = 0; s2 < GH; ++s2)
          if (s2 == s) {
            mma16816(oacc[s2][0], ah, bm[0], bm[1]);
            mma16816(oacc[s2][0], al, bm[0], bm[1]);
            mma16816(oacc[s2][1], ah, bm[2], bm[3]);
            mma16816(oacc[s2][1], al, bm[2], bm[3]);
          }
      }
    }
    __syncthreads();                              // the chunk's slot is refilled next
  }
  cp_async_wait<0>();

  // ---- partials of the split: rows gq, gq + 8; channels 128 s + cw + 8 nt + 2t + {0, 1}
  const size_t pstride = static_cast<size_t>(N) + 4;
  float* pb = a.part + ((static_cast<size_t>(b) * a.n_groups + g) * a.nq) * a.n_splits * pstride;
#pragma unroll
  for (int s = 0; s < GH; ++s)
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
      const int j = s * D + cw + 8 * nt + 2 * t;
      if (gq < a.nq) {
        float* d0 = pb + (static_cast<size_t>(gq) * a.n_splits + split) * pstride + j;
        d0[0] = oacc[s][nt][0];
        d0[1] = oacc[s][nt][1];
      }
      if (gq + 8 < a.nq) {
        float* d1 = pb + (static_cast<size_t>(gq + 8) * a.n_splits + split) * pstride + j;
        d1[0] = oacc[s][nt][2];
        d1[1] = oacc[s][nt][3];
      }
    }
  if (tid < a.nq) {
    float* d = pb + (static_cast<size_t>(tid) * a.n_splits + split) * pstride + N;
    d[0] = sm.mrow[tid];
    d[1] = sm.lrow[tid];
  }
}

// Per (query head, group, sequence), 512 threads: combine the splits (weights 2^(m_s - M)),
// o_hat_j = f^V_j O_j / l (thread = channel), then out = U_V[block rows] o_hat with four threads
// per output dim, each over a quarter of the channels.
constexpr int kGMThreads = 512;
__global__ void __launch_bounds__(kGMThreads) aatc_group_merge_kernel(const GroupDecodeArgs a) {
  extern __shared__ float msm[];                  // ohat [n], w [n_splits], part [4][128]
  float* ohat = msm;
  float* wsp = msm + a.n;
  float* psum = wsp + ((a.n_splits + 3) & ~3);
  __shared__ float red[kGMThreads / 32];
  __shared__ float s_l;
  const int i = blockIdx.x, g = blockIdx.y, b = blockIdx.z, tid = threadIdx.x;
  const int N = a.n, m = i / a.group;
  const size_t pstride = static_cast<size_t>(N) + 4;
  const float* pb = a.part + (((static_cast<size_t>(b) * a.n_groups + g) * a.nq + i) * a.n_splits) * pstride;
  // M = max_s m_s (block reduction), then w_s and l = sum_s w_s l_s
  float mloc = -INFINITY;
  for (int s2 = tid; s2 < a.n_splits; s2 += kGMThreads) mloc = fmaxf(mloc, pb[s2 * pstride + N]);
  for (int o = 16; o > 0; o >>= 1) mloc = fmaxf(mloc, __shfl_xor_sync(0xffffffffu, mloc, o));
  if ((tid & 31) == 0) red[tid >> 5] = mloc;
  __syncthreads();
  float M = -INFINITY;
  for (int w = 0; w < kGMThreads / 32; ++w) M = fmaxf(M, red[w]);
  __syncthreads();
  float lloc = 0.0f;
  for (int s2 = tid; s2 < a.n_splits; s2 += kGMThreads) {
    const float ms = pb[s2 * pstride + N];
    const float w = ms == -INFINITY ? 0.0f : exp2f(ms - M);
    wsp[s2] = w;
    lloc += w * pb[s2 * pstride + N + 1];
  }
  for (int o = 16; o > 0; o >>= 1) lloc += __shfl_xor_sync(0xffffffffu, lloc, o);
  if ((tid & 31) == 0) red[tid >> 5] = lloc;
  __syncthreads();
  if (tid == 0) {
    float l = 0.0f;
    for (int w = 0; w < kGMThreads / 32; ++w) l += red[w];
    s_l = l;
  }
  for (int j = tid; j < N; j += kGMThreads) {
    float o0 = 0.0f, o1 = 0.0f;
    int s2 = 0;
    for (; s2 + 1 < a.n_splits; s2 += 2) {
      o0 = fmaf(wsp[s2], pb[s2 * pstride + j], o0);
      o1 = fmaf(wsp[s2 + 1], pb[(s2 + 1) * pstride + j], o1);
    }
    if (s2 < a.n_splits) o0 = fmaf(wsp[s2], pb[s2 * pstride + j], o0);
    const int sl = j / D, c = j % D;
    const int slot = (a.layer * a.n_kv + g * a.gh + sl) * 2 + 1;
    ohat[j] = (o0 + o1) * a.f[slot * D + c];
  }
  __syncthreads();
  const int d = tid & (D - 1), part = tid >> 7, span = N / 4;
  const float* u = a.uvt + (static_cast<size_t>(a.layer) * a.n_groups + g) * static_cast<size_t>(N) * N +
                   static_cast<size_t>(m) * D + d;
  float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
  for (int j = part * span; j < (part + 1) * span; j += 16) {   // 16 loads in flight per thread
    float x[16];
#pragma unroll
    for (int k = 0; k < 16; ++k) x[k] = u[static_cast<size_t>(j + k) * N];
#pragma unroll
    for (int k = 0; k < 16; ++k) acc[k & 3] = fmaf(x[k], ohat[j + k], acc[k & 3]);
  }
  psum[part * D + d] = (acc[0] + acc[1]) + (acc[2] + acc[3]);
  __syncthreads();
  if (tid < D)
    a.out[(static_cast<size_t>(b) * a.n_q_heads + g * a.nq + i) * D + tid] =
        ((psum[tid] + psum[D + tid]) + (psum[2 * D + tid] + psum[3 * D + tid])) / s_l;
}

int group_splits(const Plan& plan, int batch, int n_ctx) {
  const int tiles = (n_ctx + TILE - 1) / TILE;
  const int units = batch * (plan.dims.n_kv_heads / plan.group_heads);
  return std::max(1, std::min(tiles, std::max(1, plan.num_sms) / std::max(1, units)));
}

struct GroupWs {
  size_t qf_off, part_off, bytes;
};
GroupWs group_ws_layout(const Plan& plan, int batch, int n_ctx) {
  const int ng = plan.dims.n_kv_heads / plan.group_heads, n = D * plan.group_heads;
  const int nq = plan.dims.n_q_heads / ng;
  GroupWs w;
  size_t off = (prefill_workspace(batch, plan.dims.n_kv_heads, n_ctx) + 255) / 256 * 256;
  w.qf_off = off;
  off += static_cast<size_t>(batch) * ng * nq * n * 4;
  off = (off + 255) / 256 * 256;
  w.part_off = off;
  off += static_cast<size_t>(batch) * ng * nq * group_splits(plan, batch, n_ctx) * (n + 4) * 4;
  w.bytes = off;
  return w;
}

}  // namespace

size_t group_decode_workspace(const Plan& plan, int batch, int n_ctx) { return group_ws_layout(plan, batch, n_ctx).bytes; }

cudaError_t launch_group_decode(const Plan& plan, int layer, const void* q, const void* cache, int batch, int n_ctx,
                                int max_tokens, float* out, void* ws, cudaStream_t st) {
  const int gh = plan.group_heads;
  if (gh != 2 && gh != 4) return cudaErrorNotSupported;
  const CacheGeom g = cache_geom(batch, plan.dims.n_kv_heads, max_tokens, plan.n_words);
  const GroupWs wl = group_ws_layout(plan, batch, n_ctx);
  if (plan.n_words > 32) return cudaErrorNotSupported;
  const int n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  aatc_group_codes_kernel<<<dim3(n_ctx_pad / TILE, plan.dims.n_kv_heads * 2, batch), TILE, 0, st>>>(
      static_cast<const uint32_t*>(cache), plan.dev.lay, static_cast<__half*>(ws), layer, plan.dims.n_kv_heads, n_ctx,
      n_ctx_pad, g.n_tiles, plan.n_words);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  GroupDecodeArgs a;
  a.codes = static_cast<const __half*>(ws);
  a.alpha = reinterpret_cast<const float*>(static_cast<const uint32_t*>(cache) + g.words_elems);
  a.q = static_cast<const __nv_bfloat16*>(q);
  a.uk = plan.gdev.uk;
  a.uvt = plan.gdev.uvt;
  a.f = plan.dev.f;
  a.qf = reinterpret_cast<float*>(static_cast<char*>(ws) + wl.qf_off);
  a.part = reinterpret_cast<float*>(static_cast<char*>(ws) + wl.part_off);
  a.out = out;
  a.layer = layer;
  a.n_kv = plan.dims.n_kv_heads;
  a.gh = gh;
  a.n_groups = a.n_kv / gh;
  a.group = plan.dims.n_q_heads / a.n_kv;
  a.nq = gh * a.group;
  a.n = D * gh;
  a.n_q_heads = plan.dims.n_q_heads;
  a.n_ctx = n_ctx;
  a.n_ctx_pad = (n_ctx + TILE - 1) / TILE * TILE;
  a.n_tiles = g.n_tiles;
  a.n_splits = group_splits(plan, batch, n_ctx);
  if (a.nq > 16) return cudaErrorNotSupported;
  aatc_group_query_kernel<<<dim3(a.nq, a.n_groups, batch), a.n, 0, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 grid(a.n_splits, a.n_groups, batch);
  if (gh == 2) {
    const size_t smem = sizeof(GroupAttnSmem<2>);
    e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_group_attn_kernel<2>), smem);
    if (e != cudaSuccess) return e;
    aatc_group_attn_kernel<2><<<grid, kGAThreads, smem, st>>>(a);
  } else {
    const size_t smem = sizeof(GroupAttnSmem<4>);
    e = ensure_smem_optin(reinterpret_cast<const void*>(aatc_group_attn_kernel<4>), smem);
    if (e != cudaSuccess) return e;
    aatc_group_attn_kernel<4><<<grid, kGAThreads, smem, st>>>(a);
  }
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t msm = (static_cast<size_t>(a.n) + ((a.n_splits + 3) & ~3) + 4 * D) * 4;
  aatc_group_merge_kernel<<<dim3(a.nq, a.n_groups, batch), kGMThreads, msm, st>>>(a);
  return cudaGetLastError();
}

}  // namespace aatc
