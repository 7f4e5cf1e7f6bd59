// Decode attention over head-group streams (Sec. 5 Step 1, remark on multi-head attention: the
// g_h kv-heads of a group share one transform; Def. sdpa per query head, Algorithm 1's
// reconstruct / attend / output lines in the transformed space).
//
// A group stream of n = 128 g_h channels is stored as g_h slice streams in the per-kv-head slots
// (slice s = storage channels s, s + g_h, ...), one alpha per token.  Query head j of the group
// (kv-head block m = j / group) sees the embedded query q~ (q at block m, zeros elsewhere):
//   score_t = (U_K^T q~) . h_hat_t / sqrt(128) = alpha_t sum_c q'_c f_c code_tc,
//   out     = rows of block m of U_V applied to sum_t p_t h_hat^V_t.
// Three launches per call:
//   query  per (query head, group, sequence): q'' = (U_K^T q~) f log2(e) / sqrt(128) over the n
//          slice-major channels (thread = channel)
//   attn   per (split, group, sequence), 8 warps: the slices' record words are the operands of
//          mma.sync m16n8k16 f16 (a digit or bit masked into a 16-bit half is the subnormal
//          digit 2^-24), rows = the group's <= 16 query heads: scores summed over every slice
//          and corrected by the stored-value offsets, online softmax with the exponent of
//          alpha^V folded into the running maximum (P' = 2^(s - m) alpha^V < 2), value entry sums
//          per slice, channel sums at the end of the split
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

struct GroupDecodeArgs {
  const float* alpha;        // cache alpha region [b][n_kv][K|V][n_tiles * 128]
  const __nv_bfloat16* q;    // [b][H_q][128]
  const float* uk;           // plan: U_K of every (layer, group), [n dim][n channel]
  const float* uvt;          // plan: U_V^T, [n channel][n dim]
  const float* f;            // plan: [slot][128] f_c
  float* qf;                 // workspace: folded queries [b][n_groups][nq][n]
  float* part;               // workspace: split partials [b][n_groups][nq][n_splits][n + 4]
  float* out;                // [b][H_q][128]
  const uint32_t* words;     // cache word region (the digit kernel reads the records directly)
  const short* entry;        // plan: [slot][n_entries] (channel | shift << 8), -1 padded
  const ChanEnc* enc;        // plan: [slot][128] (offset 2^(b-1) of each stored value)
  const StreamLayout* lay;   // plan: [slot]
  int layer, n_kv, gh, n_groups, group, nq, n, n_q_heads, n_ctx, n_ctx_pad, n_tiles, n_splits;
  int n_words, n_entries, ks_max, n_pairs;   // ks_max: k-steps of the widest slice; n_pairs: value tiles
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

// ---------------------------------------------------------------- digit-operand split attention
// The slices' record words are the tensor-core operands themselves (no unpacked codes): a base-4 digit (or a single bit) masked into the low bits of a 16-bit half
// is the subnormal f16 digit 2^-24, exact in the product.
//   scores: per slice and record word, k = the word's 16 D2 fields (or 16 of a D1 word's 32 bits):
//           A = q''_c 2^shift per entry (rows = queries, hi / lo), B = the 16 tokens' digits of
//           this warp (b0 = x >> 2t: fields t, t + 8; b1 = x >> 2t + 8: fields t + 4, t + 12);
//           raw = sum q'' u over all slices, s = alpha^K (raw - C) with C = sum_c q''_c 2^(b_c - 1)
//   values: per slice and 8 record entries, A = P' (queries x 16 tokens, hi / lo), B = the
//           entries' digits of those tokens from the quad-interleaved value slots; the entry sums
//           become channel sums o_c = sum_e 2^shift O_e - 2^(b_c - 1) S' (S' = the represented
//           sum of P') through shared-memory adds at the end of the split.
constexpr int kGDMaxPairs = 24;                  // value (slice, 8-entry tile) pairs per warp

struct GroupDigitSmem {
  int qfrag, pfrag, ring, oc, offs, kent, misc, total, chunk_words, kent_stride;
  __host__ __device__ GroupDigitSmem(int gh, int ks_max, int n_words, int n_entries) {
    kent_stride = (n_entries + 7) & ~7;
    int o = 0;
    qfrag = o;  o += gh * ks_max * 32 * 32;       // [slice][k-step][lane][hi, lo] uint4
    pfrag = o;  o += (TILE / 16) * 32 * 32;       // [k-step][lane][hi, lo] uint4
    chunk_words = n_words * TILE;
    ring = o;   o += kGRing * chunk_words * 4;    // record words of one slice and kind, one tile
    oc = o;     o += 16 * D * gh * 4;             // q'' of the queries in the prologue; channel sums at the end
    offs = o;   o += 2 * D * gh * 4;              // stored-value offsets 2^(b-1), keys then values
    kent = o;   o += gh * ((n_entries + 7) & ~7) * 2;   // key entry tables of the slices
    misc = o;   o += 16 * 4 * 20 + 3 * 8 * 16 * 4;
    total = o;
  }
};

template <int GH>
__global__ void __launch_bounds__(kGAThreads, 1) aatc_group_digit_kernel(const GroupDecodeArgs a) {
  constexpr int N = D * GH, NCH = 2 * GH;
  extern __shared__ __align__(128) unsigned char smb[];
  const GroupDigitSmem L(GH, a.ks_max, a.n_words, a.n_entries);
  uint4* qfrag = reinterpret_cast<uint4*>(smb + L.qfrag);
  uint4* pfrag = reinterpret_cast<uint4*>(smb + L.pfrag);
  uint32_t* ring = reinterpret_cast<uint32_t*>(smb + L.ring);
  float* oc = reinterpret_cast<float*>(smb + L.oc);
  float* qinv = reinterpret_cast<float*>(smb + L.misc);
  float* mrow = qinv + 16;
  float* lrow = mrow + 16;
  float* srow = lrow + 16;                        // S' of each query
  float* rscale = srow + 16;
  float* corr = rscale + 16;                      // C of each query
  float* redm = corr + 16;                        // [8][16]
  float* reds = redm + 8 * 16;                    // [8][16]
  float* redp = reds + 8 * 16;                    // [8][16]
  const int split = blockIdx.x, g = blockIdx.y, b = blockIdx.z;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31, gq = lane >> 2, t = lane & 3;
  const int ctx_tiles = (a.n_ctx + TILE - 1) / TILE;
  const int tile_lo = static_cast<int>(static_cast<long>(split) * ctx_tiles / a.n_splits);
  const int tile_hi = static_cast<int>(static_cast<long>(split + 1) * ctx_tiles / a.n_splits);
  const size_t slot0 = static_cast<size_t>(b) * a.n_kv + static_cast<size_t>(g) * GH;   // cache slot of slice 0
  const float* kalpha = a.alpha + (slot0 * 2) * a.n_tiles * TILE;
  const float* valpha = a.alpha + (slot0 * 2 + 1) * a.n_tiles * TILE;
  const float* qf = a.qf + (static_cast<size_t>(b) * a.n_groups + g) * a.nq * N;
  const int pslot0 = (a.layer * a.n_kv + g * GH) * 2;   // plan slot of slice 0, keys (values + 1)
  const size_t stream_words = static_cast<size_t>(a.n_tiles) * a.n_words * TILE;

  // ---- stage q'' (in the channel-sum buffer), the offsets and the key entry tables
  float* qs = oc;                                  // [16][N] q'' (rows >= nq zero)
  float* offk = reinterpret_cast<float*>(smb + L.offs);
  float* offv = offk + N;
  short* kent = reinterpret_cast<short*>(smb + L.kent);
  for (int i = tid; i < 16 * N; i += kGAThreads) qs[i] = i / N < a.nq ? qf[i] : 0.0f;
  for (int j = tid; j < N; j += kGAThreads) {
    offk[j] = a.enc[(pslot0 + 2 * (j / D)) * D + j % D].off;
    offv[j] = a.enc[(pslot0 + 2 * (j / D) + 1) * D + j % D].off;
  }
  for (int i = tid; i < GH * L.kent_stride; i += kGAThreads) {
    const int sl = i / L.kent_stride, e = i % L.kent_stride;
    kent[i] = e < a.n_entries ? a.entry[static_cast<size_t>(pslot0 + 2 * sl) * a.n_entries + e] : short(-1);
  }
  __syncthreads();
  // ---- per query (warp w: queries 2w, 2w + 1): scale bound max |q''| 2^(b-1) and C = sum q'' 2^(b-1)
#pragma unroll
  for (int h = 0; h < 2; ++h) {
    const int r = 2 * warp + h;
    float mx = 0.0f, c = 0.0f;
    for (int j = lane; j < N; j += 32) {
      const float v = qs[r * N + j], off = offk[j];
      mx = fmaxf(mx, fabsf(v) * off);              // bounds |q'' 2^shift| of every entry (shift <= b - 1)
      c = fmaf(v, off, c);
    }
    for (int o2 = 16; o2 > 0; o2 >>= 1) {
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o2));
      c += __shfl_xor_sync(0xffffffffu, c, o2);
    }
    if (lane == 0) {
      int ex = 0;
      if (mx > 0.0f) frexpf(mx, &ex);
      qinv[r] = ldexpf(1.0f, ex - 14);
      corr[r] = c;
      mrow[r] = -INFINITY;
      lrow[r] = 0.0f;
      srow[r] = 0.0f;
    }
  }
  __syncthreads();
  for (int idx = tid; idx < GH * a.ks_max * 32; idx += kGAThreads) {
    const int sl = idx / (a.ks_max * 32), ks = (idx / 32) % a.ks_max, ln = idx & 31, r0 = ln >> 2, tt = ln & 3;
    const StreamLayout& ly = a.lay[pslot0 + 2 * sl];
    const int n2 = ly.n2, ne = ly.n2 + ly.n1, n2w = n2 / 16, nks = n2w + 2 * ((ly.n1 + 31) / 32);
    int ent[4] = {-1, -1, -1, -1};                // entries in k order 2t, 2t + 1, 2t + 8, 2t + 9
    if (ks < n2w) {
      const int e = 16 * ks;
      ent[0] = e + tt; ent[1] = e + tt + 8; ent[2] = e + tt + 4; ent[3] = e + tt + 12;
    } else if (ks < nks) {
      const int u = (ks - n2w) >> 1, s2 = (ks - n2w) & 1, e = n2 + 32 * u + 8 * s2;
      ent[0] = e + tt; ent[1] = e + tt + 16; ent[2] = e + tt + 4; ent[3] = e + tt + 20;
    }
    const short* et = kent + sl * L.kent_stride;
    const float i0 = 1.0f / qinv[r0], i1 = 1.0f / qinv[r0 + 8];
    float v[8];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int ce = ent[k] >= 0 && ent[k] < ne ? et[ent[k]] : -1;
      const float w2 = ce >= 0 ? ldexpf(1.0f, (ce >> 8) & 15) : 0.0f;
      const int j = sl * D + (ce & 0xFF);
      v[2 * k] = ce >= 0 ? qs[r0 * N + j] * w2 * i0 : 0.0f;
      v[2 * k + 1] = ce >= 0 ? qs[(r0 + 8) * N + j] * w2 * i1 : 0.0f;
    }
    // A fragment: a0 = row r0 (k 2t, 2t + 1), a1 = row r0 + 8, a2 = row r0 (k 2t + 8, 2t + 9), a3 = row r0 + 8
    uint4 hi, lo;
    split2(v[0], v[2], hi.x, lo.x);
    split2(v[1], v[3], hi.y, lo.y);
    split2(v[4], v[6], hi.z, lo.z);
    split2(v[5], v[7], hi.w, lo.w);
    qfrag[((sl * a.ks_max + ks) * 32 + ln) * 2] = hi;
    qfrag[((sl * a.ks_max + ks) * 32 + ln) * 2 + 1] = lo;
  }
  __syncthreads();
  for (int i = tid; i < 16 * N; i += kGAThreads) oc[i] = 0.0f;   // q'' no longer needed

  // ---- record chunks: per tile the key words of slices 0 .. GH-1, then their value words
  const int n_chunks = (tile_hi - tile_lo) * NCH;
  const int cw = L.chunk_words;
  auto issue = [&](int u) {
    if (u < n_chunks) {
      const int tile = tile_lo + u / NCH, c = u % NCH, sl = c % GH, kind = c / GH;
      const uint32_t* src = a.words + ((slot0 + sl) * 2 + kind) * stream_words + static_cast<size_t>(tile) * cw;
      uint32_t* dst = ring + (u % kGRing) * cw;
      for (int p = tid * 4; p < cw; p += kGAThreads * 4) cp_async16(dst + p, src + p);
    }
    cp_async_commit();
  };
  for (int u = 0; u < kGRing - 1; ++u) issue(u);

  float sacc[2][4];
  float oacc[kGDMaxPairs][4];
#pragma unroll
  for (int pi = 0; pi < kGDMaxPairs; ++pi)
#pragma unroll
    for (int r = 0; r < 4; ++r) oacc[pi][r] = 0.0f;
  const int tw = 16 * warp;
  const uint32_t m2 = 0x00030003u, m1 = 0x00010001u;

  for (int u = 0; u < n_chunks; ++u) {
    issue(u + kGRing - 1);
    cp_async_wait<kGRing - 1>();
    __syncthreads();
    const int tile = tile_lo + u / NCH, c = u % NCH, sl = c % GH;
    const uint32_t* ch = ring + (u % kGRing) * cw;
    const StreamLayout ly = a.lay[pslot0 + 2 * sl + (c < GH ? 0 : 1)];
    const int n2w = ly.n2 / 16, n1w = (ly.n1 + 31) / 32;
    if (c < GH) {
      if (sl == 0)
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int r = 0; r < 4; ++r) sacc[nt][r] = 0.0f;
      const uint4* qa = qfrag + (sl * a.ks_max) * 32 * 2;
      for (int w = 0; w < n2w; ++w) {
        const uint4 ah = qa[(w * 32 + lane) * 2], al = qa[(w * 32 + lane) * 2 + 1];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
          const uint32_t x = ch[w * TILE + tw + 8 * nt + gq];
          const uint32_t b0 = (x >> (2 * t)) & m2, b1 = (x >> (2 * t + 8)) & m2;
          mma16816(sacc[nt], ah, b0, b1);
          mma16816(sacc[nt], al, b0, b1);
        }
      }
      for (int w = 0; w < n1w; ++w) {
#pragma unroll
        for (int s2 = 0; s2 < 2; ++s2) {
          const int ks = n2w + 2 * w + s2;
          const uint4 ah = qa[(ks * 32 + lane) * 2], al = qa[(ks * 32 + lane) * 2 + 1];
#pragma unroll
          for (int nt = 0; nt < 2; ++nt) {
            const uint32_t x = ch[(n2w + w) * TILE + tw + 8 * nt + gq];
            const uint32_t b0 = (x >> (t + 8 * s2)) & m1, b1 = (x >> (t + 4 + 8 * s2)) & m1;
            mma16816(sacc[nt], ah, b0, b1);
            mma16816(sacc[nt], al, b0, b1);
          }
        }
      }
      if (sl == GH - 1) {
        // ---- online softmax of the tile, raw = acc 2^24 / scale - C.  Lane (gq, t) holds rows gq,
        // gq + 8 and tokens tw + 8 nt + 2t + {0, 1}; e = s + floor(log2 alpha^V) keeps
        // P' = 2^(e - m) mant(alpha^V) < 2.
        float e[2][4], mant[2][4], lav[2][4];
        float mx0 = -INFINITY, mx1 = -INFINITY;
        const float q0 = qinv[gq] * 16777216.0f, q1 = qinv[gq + 8] * 16777216.0f;
        const float c0 = corr[gq], c1 = corr[gq + 8];
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
              const float sv = (r < 2 ? fmaf(sacc[nt][r], q0, -c0) : fmaf(sacc[nt][r], q1, -c1)) * ak;
              int ex = 0;
              const float fr = frexpf(avv, &ex);
              lv = avv > 0.0f ? static_cast<float>(max(ex - 1, -64)) : -64.0f;
              mv = avv > 0.0f ? fr * 2.0f : 0.0f;
              if (avv > 0.0f && ex - 1 < -64) mv = avv * 18446744073709551616.0f;
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
          redm[warp * 16 + gq] = mx0;
          redm[warp * 16 + gq + 8] = mx1;
        }
        __syncthreads();
        if (tid < 16) {
          float mt = -INFINITY;
#pragma unroll
          for (int w = 0; w < 8; ++w) mt = fmaxf(mt, redm[w * 16 + tid]);
          const float mo = mrow[tid], mn = fmaxf(mo, mt);
          rscale[tid] = mo == -INFINITY ? 0.0f : fexp2(mo - mn);
          mrow[tid] = mn;
        }
        __syncthreads();
        const float m0 = mrow[gq], m1r = mrow[gq + 8];
        float ls0 = 0.0f, ls1 = 0.0f, ps0 = 0.0f, ps1 = 0.0f;
        float p[2][4];
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
          for (int r = 0; r < 4; ++r) {
            const float mm = r < 2 ? m0 : m1r;
            const float x = e[nt][r] == -INFINITY ? 0.0f : fexp2(e[nt][r] - mm);
            p[nt][r] = x * mant[nt][r];
            const float l = e[nt][r] == -INFINITY ? 0.0f : x * exp2f(-lav[nt][r]);
            if (r < 2) ls0 += l;
            else ls1 += l;
          }
        uint4 ph, pl;
        split2(p[0][0], p[0][1], ph.x, pl.x);
        split2(p[0][2], p[0][3], ph.y, pl.y);
        split2(p[1][0], p[1][1], ph.z, pl.z);
        split2(p[1][2], p[1][3], ph.w, pl.w);
        pfrag[(warp * 32 + lane) * 2] = ph;
        pfrag[(warp * 32 + lane) * 2 + 1] = pl;
        // S': the represented P' (hi + lo) that the value MMAs add
        {
          const __half2* hh = reinterpret_cast<const __half2*>(&ph);
          const __half2* ll = reinterpret_cast<const __half2*>(&pl);
          float2 v;
          v = __half22float2(hh[0]); ps0 += v.x + v.y; v = __half22float2(ll[0]); ps0 += v.x + v.y;
          v = __half22float2(hh[2]); ps0 += v.x + v.y; v = __half22float2(ll[2]); ps0 += v.x + v.y;
          v = __half22float2(hh[1]); ps1 += v.x + v.y; v = __half22float2(ll[1]); ps1 += v.x + v.y;
          v = __half22float2(hh[3]); ps1 += v.x + v.y; v = __half22float2(ll[3]); ps1 += v.x + v.y;
        }
        ls0 += __shfl_xor_sync(0xffffffffu, ls0, 1);
        ls0 += __shfl_xor_sync(0xffffffffu, ls0, 2);
        ls1 += __shfl_xor_sync(0xffffffffu, ls1, 1);
        ls1 += __shfl_xor_sync(0xffffffffu, ls1, 2);
        ps0 += __shfl_xor_sync(0xffffffffu, ps0, 1);
        ps0 += __shfl_xor_sync(0xffffffffu, ps0, 2);
        ps1 += __shfl_xor_sync(0xffffffffu, ps1, 1);
        ps1 += __shfl_xor_sync(0xffffffffu, ps1, 2);
        if (t == 0) {
          reds[warp * 16 + gq] = ls0;
          reds[warp * 16 + gq + 8] = ls1;
          redp[warp * 16 + gq] = ps0;
          redp[warp * 16 + gq + 8] = ps1;
        }
        // value accumulators: rows of D are the queries (c0, c1: row gq; c2, c3: row gq + 8)
        const float r0 = rscale[gq], r1 = rscale[gq + 8];
#pragma unroll
        for (int pi = 0; pi < kGDMaxPairs; ++pi) {
          oacc[pi][0] *= r0;
          oacc[pi][1] *= r0;
          oacc[pi][2] *= r1;
          oacc[pi][3] *= r1;
        }
        __syncthreads();
        if (tid < 16) {
          float lt = 0.0f, pt = 0.0f;
#pragma unroll
          for (int w = 0; w < 8; ++w) {
            lt += reds[w * 16 + tid];
            pt += redp[w * 16 + tid];
          }
          lrow[tid] = lrow[tid] * rscale[tid] + lt;
          srow[tid] = srow[tid] * rscale[tid] + pt;
        }
      }
    } else {
      // ---- O_e += P' . digit_e for this warp's (slice, 8-entry tile) pairs of slice sl
      const int ne = ly.n2 + ly.n1;
#pragma unroll
      for (int pi = 0; pi < kGDMaxPairs; ++pi) {
        const int pr = warp + 8 * pi;
        if (pr >= a.n_pairs) break;
        // pairs are numbered slice-major: pr = sl' * ntp + nt with ntp n-tiles per slice
        const int ntp = (a.ks_max * 16 + 7) / 8;
        const int p_sl = pr / ntp, p_nt = pr % ntp;
        if (p_sl != sl) continue;
        const int e = 8 * p_nt + gq;               // this lane's entry (B column gq)
        uint32_t widx = 0, shb = 0, msk = 0;
        int qpos = 0;
        if (e < ly.n2) {
          const int f = e & 15;
          widx = e >> 4;
          qpos = (f >> 2) == 1 ? 2 : (f >> 2) == 2 ? 1 : (f >> 2);
          shb = 2 * (f & 3);
          msk = 3u;
        } else if (e < ne) {
          const int e1 = e - ly.n2, bb = e1 & 31;
          widx = n2w + (e1 >> 5);
          qpos = (bb >> 3) == 1 ? 2 : (bb >> 3) == 2 ? 1 : (bb >> 3);
          shb = bb & 7;
          msk = 1u;
        }
        const uint32_t mlo = msk, mhi = msk << 16;
        const uint32_t* wr = ch + widx * TILE + qpos;
        const int i0 = 2 * (t & 1);
#pragma unroll
        for (int kt = 0; kt < TILE / 16; ++kt) {
          const uint32_t x0 = wr[4 * (4 * kt + (t >> 1))], x1 = wr[4 * (4 * kt + 2 + (t >> 1))];
          const uint32_t y0 = x0 >> (8 * i0 + shb), y1 = x1 >> (8 * i0 + shb);
          const uint32_t b0 = (y0 & mlo) | ((y0 << 8) & mhi), b1 = (y1 & mlo) | ((y1 << 8) & mhi);
          const uint4 ah = pfrag[(kt * 32 + lane) * 2], al = pfrag[(kt * 32 + lane) * 2 + 1];
          mma16816(oacc[pi], ah, b0, b1);
          mma16816(oacc[pi], al, b0, b1);
        }
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();

  // ---- entry sums -> channel sums (shared-memory adds), then the split's partials
  {
    const int ntp = (a.ks_max * 16 + 7) / 8;
#pragma unroll
    for (int pi = 0; pi < kGDMaxPairs; ++pi) {
      const int pr = warp + 8 * pi;
      if (pr >= a.n_pairs) break;
      const int p_sl = pr / ntp, p_nt = pr % ntp;
      const short* et = a.entry + static_cast<size_t>(pslot0 + 2 * p_sl + 1) * a.n_entries;
      const StreamLayout ly = a.lay[pslot0 + 2 * p_sl + 1];
#pragma unroll
      for (int k = 0; k < 2; ++k) {
        const int e = 8 * p_nt + 2 * t + k;        // D column 2t + k
        const int ce = e < ly.n2 + ly.n1 ? et[e] : -1;
        if (ce < 0) continue;
        const float w2 = ldexpf(1.0f, ((ce >> 8) & 15) + 24);   // digits entered as d 2^-24
        const int j = p_sl * D + (ce & 0xFF);
        if (gq < a.nq) atomicAdd(&oc[gq * N + j], w2 * oacc[pi][k]);
        if (gq + 8 < a.nq) atomicAdd(&oc[(gq + 8) * N + j], w2 * oacc[pi][2 + k]);
      }
    }
  }
  __syncthreads();
  const size_t pstride = static_cast<size_t>(N) + 4;
  float* pb = a.part + ((static_cast<size_t>(b) * a.n_groups + g) * a.nq) * a.n_splits * pstride;
  for (int idx = tid; idx < a.nq * N; idx += kGAThreads) {
    const int i = idx / N, j = idx % N;
    pb[(static_cast<size_t>(i) * a.n_splits + split) * pstride + j] = oc[i * N + j] - offv[j] * srow[i];
  }
  if (tid < a.nq) {
    float* d = pb + (static_cast<size_t>(tid) * a.n_splits + split) * pstride + N;
    d[0] = mrow[tid];
    d[1] = lrow[tid];
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
// k-steps (D2 words + 2 x D1 words) of the widest slice stream of `layer` (keys or values)
int group_ks_max(const Plan& plan, int layer) {
  int m = 1;
  for (int h = 0; h < plan.dims.n_kv_heads; ++h)
    for (int kind = 0; kind < 2; ++kind) {
      const StreamLayout& ly = plan.layout[(layer * plan.dims.n_kv_heads + h) * 2 + kind];
      m = std::max(m, ly.n2 / 16 + 2 * ((ly.n1 + 31) / 32));
    }
  return m;
}

GroupWs group_ws_layout(const Plan& plan, int batch, int n_ctx) {
  const int ng = plan.dims.n_kv_heads / plan.group_heads, n = D * plan.group_heads;
  const int nq = plan.dims.n_q_heads / ng;
  GroupWs w;
  size_t off = 0;
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
  GroupDecodeArgs a;
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
  a.words = static_cast<const uint32_t*>(cache);
  a.entry = plan.dev.entry;
  a.enc = plan.dev.enc;
  a.lay = plan.dev.lay;
  a.n_words = plan.n_words;
  a.n_entries = plan.n_entries;
  a.ks_max = group_ks_max(plan, layer);
  a.n_pairs = gh * 2 * a.ks_max;                 // (slice, 8-entry tile) pairs of the value records
  if (a.nq > 16 || a.n_pairs > 8 * kGDMaxPairs) return cudaErrorNotSupported;
  aatc_group_query_kernel<<<dim3(a.nq, a.n_groups, batch), a.n, 0, st>>>(a);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const dim3 grid(a.n_splits, a.n_groups, batch);
  const size_t smem = static_cast<size_t>(GroupDigitSmem(gh, a.ks_max, a.n_words, a.n_entries).total);
  if (smem > 227 * 1024) return cudaErrorNotSupported;
  const void* kern = gh == 2 ? reinterpret_cast<const void*>(aatc_group_digit_kernel<2>)
                             : reinterpret_cast<const void*>(aatc_group_digit_kernel<4>);
  e = ensure_smem_optin(kern, smem);
  if (e != cudaSuccess) return e;
  if (gh == 2) aatc_group_digit_kernel<2><<<grid, kGAThreads, smem, st>>>(a);
  else aatc_group_digit_kernel<4><<<grid, kGAThreads, smem, st>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  const size_t msm = (static_cast<size_t>(a.n) + ((a.n_splits + 3) & ~3) + 4 * D) * 4;
  aatc_group_merge_kernel<<<dim3(a.nq, a.n_groups, batch), kGMThreads, msm, st>>>(a);
  return cudaGetLastError();
}

}  // namespace aatc
